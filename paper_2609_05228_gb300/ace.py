"""ctypes binding of libace.so (include/ace.h). Argument marshalling only:
every step of the layer runs in the library's CUDA kernels.

Functions keep the C names. Device pointers may be given as ints or as torch
tensors (their data_ptr()); host outputs are returned as numpy arrays.
Streams may be None (default stream), an int handle or a torch.cuda.Stream.
The library is loaded on first use; a missing library raises AceError.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_LIBDIR = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_lib")
# ACE_LIB_VARIANT=debug loads libace_debug.so (index guards and canary words)
LIBNAME = "libace_debug.so" if os.environ.get("ACE_LIB_VARIANT") == "debug" else "libace.so"
LIBPATH = os.path.join(_LIBDIR, LIBNAME)

ACE_BF16, ACE_F32 = 0, 1
ACE_SKIP_THRESHOLD, ACE_SKIP_RATIO = 0, 1
# Skip rules (ace_fusion): index = enum value. "max" is ACE.
FUSIONS = ("max", "min", "mean", "gsp", "rcr", "score")
ACE_FUSION_MAX, ACE_FUSION_MIN, ACE_FUSION_MEAN, ACE_FUSION_GSP, ACE_FUSION_RCR, ACE_FUSION_SCORE = range(6)
STATUS = {0: "ACE_OK", 1: "ACE_ERR_INVALID_ARG", 2: "ACE_ERR_UNSUPPORTED", 3: "ACE_ERR_OOM",
          4: "ACE_ERR_CUDA", 5: "ACE_ERR_TIMEOUT", 6: "ACE_ERR_NUMERIC", 7: "ACE_ERR_STATE"}


class AceError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{STATUS.get(status, status)}: {msg}")
        self.status = status


class ace_layer_desc(ctypes.Structure):
    _fields_ = [("hidden", ctypes.c_int), ("n_experts", ctypes.c_int), ("top_k", ctypes.c_int),
                ("ffn", ctypes.c_int), ("max_tokens", ctypes.c_int), ("dtype", ctypes.c_int),
                ("eps", ctypes.c_float), ("rms_eps", ctypes.c_float), ("router_temp", ctypes.c_float),
                ("min_active", ctypes.c_int), ("has_router_bias", ctypes.c_int), ("add_residual", ctypes.c_int)]


class ace_skip_ctl(ctypes.Structure):
    _fields_ = [("mode", ctypes.c_int), ("value", ctypes.c_float), ("fusion", ctypes.c_int)]


_lib = None
_P = ctypes.c_void_p
_I = ctypes.c_int
_S = ctypes.c_int  # ace_status


def lib() -> ctypes.CDLL:
    """Load libace.so (raises AceError if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIBPATH):
            raise AceError(4, f"{LIBNAME} not found at {LIBPATH}; build it with "
                              "`python -m paper_2609_05228_gb300.build`")
        L = ctypes.CDLL(LIBPATH)
        sig = {
            "ace_layer_create": (_S, [ctypes.POINTER(ace_layer_desc), _P, _P, _P, _P, _P, _P, _P, _P, _P,
                                      ctypes.POINTER(_P)]),
            "ace_layer_destroy": (None, [_P]),
            "ace_moe_forward": (_S, [_P, _P, _P, _I, ace_skip_ctl, _P]),
            "ace_moe_forward_host": (_S, [_P, _P, _P, _I, ace_skip_ctl, _P]),
            "ace_route_logits": (_S, [_P, _P, _I, ace_skip_ctl, _P]),
            "ace_last_skip_mask": (_S, [_P, _P, _P, _P, _P, _P]),
            "ace_last_router_logits": (_S, [_P, _P]),
            "ace_last_permutation": (_S, [_P, _P, _P]),
            "ace_layer_sync": (_S, [_P]),
            "ace_debug_exp32": (_S, [_P, _P, _I, _P]),
            "ace_debug_set_wait_budget": (_S, [_P, ctypes.c_longlong]),
            "ace_debug_checks_enabled": (_I, []),
            "ace_debug_poke_canary": (_S, [_P, _I]),
            "ace_layer_get_desc": (_S, [_P, ctypes.POINTER(ace_layer_desc)]),
            "ace_layer_set_profiling": (_S, [_P, _I]),
            "ace_last_stage_times": (_S, [_P, _P, _I, _P]),
            "ace_last_launch_count": (_S, [_P, _P]),
            "ace_route_decide_noalloc": (_S, [_P, _I, _I, _I, _P, _P, ctypes.c_float, _I, ace_skip_ctl, _P, _P, _P,
                                              _P, _P]),
            "ace_stack_create": (_S, [ctypes.POINTER(_P), _I, ctypes.POINTER(_P)]),
            "ace_stack_forward": (_S, [_P, _P, _P, _I, ace_skip_ctl, _P]),
            "ace_stack_destroy": (None, [_P]),
            "ace_stack_forward_host": (_S, [_P, _P, _P, _I, ace_skip_ctl, _P]),
            "ace_offline_tables_device": (_S, [_I, _I, _I, _P, _P, _P, _P, _P, ctypes.c_double, _I, ctypes.c_size_t,
                                               _P, _P, _P]),
            "ace_status_string": (ctypes.c_char_p, [_S]),
            "ace_last_error_message": (ctypes.c_char_p, []),
        }
        for name, (res, args) in sig.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def _ptr(x) -> int | None:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    if isinstance(x, np.ndarray):
        return x.ctypes.data
    raise TypeError(f"cannot take a pointer of {type(x)}")


def _stream(s) -> int | None:
    if s is None:
        return None
    if isinstance(s, int):
        return s
    return s.cuda_stream


def _check(st: int) -> None:
    if st != 0:
        raise AceError(st, lib().ace_last_error_message().decode())


def _fusion(fusion) -> int:
    if isinstance(fusion, str):
        if fusion not in FUSIONS:
            raise ValueError(f"unknown fusion {fusion!r}; one of {FUSIONS}")
        return FUSIONS.index(fusion)
    return int(fusion)


def _ctl(mode, value, fusion=ACE_FUSION_MAX) -> ace_skip_ctl:
    if isinstance(mode, str):
        mode = ACE_SKIP_RATIO if mode == "ratio" else ACE_SKIP_THRESHOLD
    return ace_skip_ctl(int(mode), float(value), _fusion(fusion))


def ace_layer_create(desc: ace_layer_desc, router_w, router_b, w_gate, w_up, w_down, rms_gamma,
                     a_gsp: np.ndarray, a_rcr: np.ndarray, stream=None) -> int:
    a_gsp = np.ascontiguousarray(a_gsp, dtype=np.float32)
    a_rcr = np.ascontiguousarray(a_rcr, dtype=np.float32)
    out = _P()
    _check(lib().ace_layer_create(ctypes.byref(desc), _ptr(router_w), _ptr(router_b), _ptr(w_gate),
                                  _ptr(w_up), _ptr(w_down), _ptr(rms_gamma), a_gsp.ctypes.data,
                                  a_rcr.ctypes.data, _stream(stream), ctypes.byref(out)))
    return out.value


def ace_layer_destroy(layer: int) -> None:
    if layer:
        lib().ace_layer_destroy(layer)


def ace_moe_forward(layer: int, x, out, T: int, mode, value: float, stream=None, fusion=ACE_FUSION_MAX) -> None:
    _check(lib().ace_moe_forward(layer, _ptr(x), _ptr(out), int(T), _ctl(mode, value, fusion), _stream(stream)))


def ace_moe_forward_host(layer: int, x_host, out_host, T: int, mode, value: float, stream=None, fusion=ACE_FUSION_MAX) -> None:
    _check(lib().ace_moe_forward_host(layer, _ptr(x_host), _ptr(out_host), int(T), _ctl(mode, value, fusion),
                                      _stream(stream)))


def ace_route_logits(layer: int, logits, T: int, mode, value: float, stream=None, fusion=ACE_FUSION_MAX) -> None:
    _check(lib().ace_route_logits(layer, _ptr(logits), int(T), _ctl(mode, value, fusion), _stream(stream)))


def ace_stack_create(layers) -> int:
    """A stack over layer handles (ints); the layers must outlive it."""
    arr = (_P * len(layers))(*[int(h) for h in layers])
    out = _P()
    _check(lib().ace_stack_create(arr, len(layers), ctypes.byref(out)))
    return out.value


def ace_stack_forward(stack: int, x, out, T: int, mode, value: float, stream=None, fusion=ACE_FUSION_MAX) -> None:
    _check(lib().ace_stack_forward(stack, _ptr(x), _ptr(out), int(T), _ctl(mode, value, fusion), _stream(stream)))


def ace_stack_forward_host(stack: int, x_host, out_host, T: int, mode, value: float, stream=None,
                           fusion=ACE_FUSION_MAX) -> None:
    _check(lib().ace_stack_forward_host(stack, _ptr(x_host), _ptr(out_host), int(T), _ctl(mode, value, fusion),
                                        _stream(stream)))


def ace_stack_destroy(stack: int) -> None:
    if stack:
        lib().ace_stack_destroy(stack)


def ace_last_skip_mask(layer: int, T: int, k: int):
    """Returns (skip uint8 [T,k], ids int32 [T,k], gates_hat float32 [T,k], tau, R)."""
    skip = np.zeros((T, k), np.uint8)
    ids = np.zeros((T, k), np.int32)
    gh = np.zeros((T, k), np.float32)
    tau = np.zeros(1, np.float32)
    r = np.zeros(1, np.int32)
    _check(lib().ace_last_skip_mask(layer, skip.ctypes.data, ids.ctypes.data, gh.ctypes.data,
                                    tau.ctypes.data, r.ctypes.data))
    return skip, ids, gh, tau[0], int(r[0])


def ace_last_router_logits(layer: int, T: int, N: int) -> np.ndarray:
    z = np.zeros((T, N), np.float32)
    _check(lib().ace_last_router_logits(layer, z.ctypes.data))
    return z


def ace_last_permutation(layer: int, N: int, R: int):
    off = np.zeros(N + 1, np.int32)
    perm = np.zeros(max(R, 1), np.int32)
    _check(lib().ace_last_permutation(layer, off.ctypes.data, perm.ctypes.data))
    return off, perm[:R]


def ace_layer_sync(layer: int) -> None:
    _check(lib().ace_layer_sync(layer))


def ace_debug_set_wait_budget(layer: int, cycles: int) -> None:
    _check(lib().ace_debug_set_wait_budget(layer, int(cycles)))


def ace_debug_checks_enabled() -> bool:
    return bool(lib().ace_debug_checks_enabled())


def ace_debug_poke_canary(layer: int, index: int) -> None:
    _check(lib().ace_debug_poke_canary(layer, int(index)))


def ace_debug_exp32(x, y, n: int, stream=None) -> None:
    _check(lib().ace_debug_exp32(_ptr(x), _ptr(y), int(n), _stream(stream)))


STAGES = ["rmsnorm", "router", "route", "gather", "gate_up", "down", "combine"]


def ace_layer_set_profiling(layer: int, enable: bool) -> None:
    _check(lib().ace_layer_set_profiling(layer, int(bool(enable))))


def ace_last_stage_times(layer: int) -> dict:
    ms = np.zeros(16, np.float32)
    n = np.zeros(1, np.int32)
    _check(lib().ace_last_stage_times(layer, ms.ctypes.data, 16, n.ctypes.data))
    return {STAGES[i] if i < len(STAGES) else f"stage{i}": float(ms[i]) for i in range(int(n[0]))}


def ace_route_decide_noalloc(logits, T: int, n_experts: int, top_k: int, a_gsp, a_rcr, eps: float,
                             min_active: int, mode, value: float, ids, skip, gates_hat, tau, stream=None,
                             fusion=ACE_FUSION_MAX) -> None:
    """Routing decision without a layer or any device allocation (all pointers are device buffers)."""
    _check(lib().ace_route_decide_noalloc(_ptr(logits), int(T), int(n_experts), int(top_k), _ptr(a_gsp), _ptr(a_rcr),
                                          float(eps), int(min_active), _ctl(mode, value, fusion), _ptr(ids), _ptr(skip),
                                          _ptr(gates_hat), _ptr(tau), _stream(stream)))


def ace_offline_tables_device(d: int, N: int, m: int, gamma, router_w, w_gate, w_up, w_down, eps: float = 1e-6,
                              rcr_apply_gamma: bool = False, tile_budget: int = 0, stream=None):
    """(A^GSP, A^RCR) float32 [N] computed on the GPU from bf16 device weights."""
    gsp = np.empty(N, np.float32)
    rcr = np.empty(N, np.float32)
    _check(lib().ace_offline_tables_device(int(d), int(N), int(m), _ptr(gamma), _ptr(router_w), _ptr(w_gate),
                                           _ptr(w_up), _ptr(w_down), float(eps), int(bool(rcr_apply_gamma)),
                                           int(tile_budget), gsp.ctypes.data, rcr.ctypes.data, _stream(stream)))
    return gsp, rcr


def ace_last_launch_count(layer: int) -> int:
    n = np.zeros(1, np.int32)
    _check(lib().ace_last_launch_count(layer, n.ctypes.data))
    return int(n[0])


def ace_layer_get_desc(layer: int) -> ace_layer_desc:
    d = ace_layer_desc()
    _check(lib().ace_layer_get_desc(layer, ctypes.byref(d)))
    return d


# --------------------------------------------------------------------------
# Convenience: a layer built from host arrays (synth.LayerWeights-like), with
# torch used only to hold the device copies during creation.
# --------------------------------------------------------------------------

class AceLayer:
    """Owns one ace_layer. `w` holds nn.Linear-shaped host arrays (bf16 as
    uint16 bits or float32); a_gsp / a_rcr are the offline tables."""

    def __init__(self, w, a_gsp, a_rcr, max_tokens: int, device: int = 0, residual: bool = False):
        import torch

        spec = w.spec
        bf = spec.dtype == "bf16"
        tdt = torch.bfloat16 if bf else torch.float32
        dev = torch.device("cuda", device)

        def up(a):
            a = np.ascontiguousarray(a)
            if a.dtype == np.uint16:
                return torch.from_numpy(a.view(np.int16)).view(torch.bfloat16).to(dev)
            return torch.from_numpy(a.astype(np.float32, copy=False)).to(dev)

        has_bias = bool(np.any(w.router_b != 0))
        self.desc = ace_layer_desc(spec.hidden, spec.n_experts, spec.top_k, spec.ffn, int(max_tokens),
                                   ACE_BF16 if bf else ACE_F32, spec.eps, spec.rms_eps, spec.router_temp,
                                   spec.min_active, int(has_bias), int(residual))
        tensors = [up(w.router_w), torch.from_numpy(np.ascontiguousarray(w.router_b, np.float32)).to(dev),
                   up(w.w_gate), up(w.w_up), up(w.w_down), up(w.gamma)]
        torch.cuda.synchronize(dev)
        self.handle = ace_layer_create(self.desc, *tensors, a_gsp, a_rcr)
        del tensors
        self.spec = spec
        self.torch_dtype = tdt

    def forward(self, x, out, T: int, mode="threshold", value: float = 0.0, stream=None,
                fusion=ACE_FUSION_MAX) -> None:
        ace_moe_forward(self.handle, x, out, T, mode, value, stream, fusion)

    def close(self) -> None:
        if getattr(self, "handle", None):
            ace_layer_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
