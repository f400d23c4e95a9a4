"""ctypes binding of libec2moe.so (the C ABI in include/ec2moe.h).

Argument marshalling only: every function passes device addresses, sizes and
the stream handle straight to the C entry point of the same name and raises
``Ec2moeError`` when it returns a status other than EC2MOE_OK.  There is no
fallback: if the library is missing, ``load()`` raises.

Tensors may be torch tensors (their ``data_ptr()`` is passed), plain integer
addresses, or None (NULL).  ``stream`` may be a ``torch.cuda.Stream``, an
integer cudaStream_t, or None for torch's current stream on the current device.
"""

from __future__ import annotations

import ctypes
import os
from typing import Optional

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "libec2moe.so")

OK = 0
ERR_INVALID_ARG = 1
ERR_ALL_MASKED = 2
ERR_TOO_FEW_EXPERTS = 3
ERR_UNSUPPORTED = 4
ERR_CUDA = 5
ERR_TIMEOUT = 6
ERR_WORKSPACE = 7
ERR_MISALIGNED = 8

F32 = 0
BF16 = 1
GELU = 0
SWIGLU = 1

EXPORTED = [
    "ec2moe_workspace_size", "ec2moe_experts_workspace_size", "ec2moe_route_workspace_size",
    "ec2moe_gate", "ec2moe_route", "ec2moe_experts", "ec2moe_shared_experts", "ec2moe_combine",
    "ec2moe_lr_encode", "ec2moe_lr_decode", "ec2moe_layer_forward", "ec2moe_last_device_error",
    "ec2moe_last_launch_count", "ec2moe_status_string", "ec2moe_profile_enable", "ec2moe_profile_count",
    "ec2moe_profile_read", "ec2moe_profile_reset", "ec2moe_route_noalloc", "ec2moe_set_wait_budget",
    "ec2moe_get_wait_budget", "ec2moe_schedule", "ec2moe_schedule_objective", "ec2moe_expert_tasks",
    "ec2moe_pipelined_workspace_size", "ec2moe_layer_forward_pipelined", "ec2moe_profile_only",
]

END = 0
CLOUD = 1


class LayerDesc(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in
                ("T", "d", "E", "d_ff", "k", "n_groups", "act", "dtype", "r", "n_shared", "d_ff_shared",
                 "renorm_topk", "top_groups")]


class LayerWeights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in
                ("W_local", "b_local", "W_global", "b_global", "W1", "W3", "W2", "W1s", "W3s", "W2s",
                 "V_enc", "V_dec")]


class Ec2moeError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} (status {status})")


_lib: Optional[ctypes.CDLL] = None

_P = ctypes.c_void_p
_D = ctypes.POINTER(LayerDesc)
_SIGS = {
    "ec2moe_workspace_size": (ctypes.c_size_t, [_D]),
    "ec2moe_experts_workspace_size": (ctypes.c_size_t, [_D]),
    "ec2moe_route_workspace_size": (ctypes.c_size_t, [_D]),
    "ec2moe_gate": (ctypes.c_int, [_D, _P, _P, _P, _P, _P, _P, _P, _P, _P]),
    "ec2moe_route": (ctypes.c_int, [_D, _P, _P, _P, _P, _P, _P, ctypes.c_int32, _P, _P, ctypes.c_size_t, _P]),
    "ec2moe_route_noalloc": (ctypes.c_int, [_D, _P, _P, _P, _P, _P, _P, ctypes.c_int32, _P, _P]),
    "ec2moe_experts": (ctypes.c_int, [_D, _P, _P, _P, _P, _P, _P, _P, _P, _P, ctypes.c_size_t, _P]),
    "ec2moe_shared_experts": (ctypes.c_int, [_D, _P, _P, _P, _P, _P, _P, ctypes.c_size_t, _P]),
    "ec2moe_combine": (ctypes.c_int, [_D, _P, _P, _P, _P]),
    "ec2moe_lr_encode": (ctypes.c_int, [_D, _P, _P, _P, _P]),
    "ec2moe_lr_decode": (ctypes.c_int, [_D, _P, _P, _P, _P]),
    "ec2moe_layer_forward": (ctypes.c_int, [_D, ctypes.POINTER(LayerWeights), _P, _P, _P, _P, _P, _P, _P, _P,
                                            ctypes.c_size_t, _P]),
    "ec2moe_last_device_error": (ctypes.c_int, [_P]),
    "ec2moe_last_launch_count": (ctypes.c_int32, []),
    "ec2moe_status_string": (ctypes.c_char_p, [ctypes.c_int]),
    "ec2moe_profile_enable": (ctypes.c_int, [ctypes.c_int32]),
    "ec2moe_profile_count": (ctypes.c_int32, []),
    "ec2moe_profile_only": (ctypes.c_int, [ctypes.c_int32]),
    "ec2moe_profile_read": (ctypes.c_int, [ctypes.c_int32, ctypes.POINTER(ctypes.c_char_p),
                                           ctypes.POINTER(ctypes.c_float)]),
    "ec2moe_profile_reset": (None, []),
    "ec2moe_set_wait_budget": (ctypes.c_int, [ctypes.c_int64]),
    "ec2moe_get_wait_budget": (ctypes.c_int64, []),
    "ec2moe_schedule": (ctypes.c_int, [ctypes.c_int32, _P, _P, ctypes.c_double, ctypes.c_double, ctypes.c_double,
                                       ctypes.c_double, ctypes.c_double, _P, _P, _P, _P]),
    "ec2moe_schedule_objective": (ctypes.c_int, [ctypes.c_int32, _P, _P, _P, ctypes.c_double, ctypes.c_double,
                                                 ctypes.c_double, _P]),
    "ec2moe_expert_tasks": (ctypes.c_int, [_D, _P, _P, _P, _P, _P]),
    "ec2moe_pipelined_workspace_size": (ctypes.c_size_t, [_D, ctypes.c_int32]),
    "ec2moe_layer_forward_pipelined": (ctypes.c_int, [_D, ctypes.POINTER(LayerWeights), _P, _P, _P, _P, _P, _P, _P,
                                                      _P, ctypes.c_size_t, ctypes.c_int32, _P, _P]),
}


def load() -> ctypes.CDLL:
    """Load libec2moe.so from the package directory (build it first with build.build())."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                               "`python -m paper_2508_06024_gb300.build`")
        lib = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _mask(mask):
    if mask is None or isinstance(mask, ctypes.Array):
        return mask
    vals = [int(v) for v in (mask.tolist() if hasattr(mask, "tolist") else mask)]
    return (ctypes.c_uint8 * len(vals))(*vals)


def _dref(desc):
    return None if desc is None else ctypes.byref(desc)


def _check(status: int, where: str) -> None:
    if status != OK:
        raise Ec2moeError(status, where)


def status_string(status: int) -> str:
    return load().ec2moe_status_string(status).decode()


def make_desc(T, d, E, d_ff, k, n_groups=1, act=GELU, dtype=BF16, r=0, n_shared=0, d_ff_shared=0,
              renorm_topk=0, top_groups=0) -> LayerDesc:
    return LayerDesc(T, d, E, d_ff, k, n_groups, act, dtype, r, n_shared, d_ff_shared, renorm_topk, top_groups)


def host_mask(mask):
    """A reusable host uint8 array for the ``mask`` argument (saves per-call marshalling)."""
    return _mask(mask)


def make_weights(W_local=None, b_local=None, W_global=None, b_global=None, W1=None, W3=None, W2=None,
                 W1s=None, W3s=None, W2s=None, V_enc=None, V_dec=None) -> LayerWeights:
    return LayerWeights(*(_ptr(t) for t in (W_local, b_local, W_global, b_global, W1, W3, W2, W1s, W3s, W2s,
                                            V_enc, V_dec)))


def ec2moe_workspace_size(desc: LayerDesc) -> int:
    return int(load().ec2moe_workspace_size(_dref(desc)))


def ec2moe_experts_workspace_size(desc: LayerDesc) -> int:
    return int(load().ec2moe_experts_workspace_size(_dref(desc)))


def ec2moe_route_workspace_size(desc: LayerDesc) -> int:
    return int(load().ec2moe_route_workspace_size(_dref(desc)))


def ec2moe_gate(desc, X, W_local, b_local, W_global, b_global, mask, topk_idx, topk_w, stream=None):
    _check(load().ec2moe_gate(_dref(desc), _ptr(X), _ptr(W_local), _ptr(b_local), _ptr(W_global),
                              _ptr(b_global), _mask(mask), _ptr(topk_idx), _ptr(topk_w), _stream(stream)),
           "ec2moe_gate")


def ec2moe_route(desc, topk_idx, counts, offsets, perm, inv_perm=None, src=None, width=0, dst=None,
                 workspace=None, ws_bytes=0, stream=None):
    _check(load().ec2moe_route(_dref(desc), _ptr(topk_idx), _ptr(counts), _ptr(offsets), _ptr(perm),
                               _ptr(inv_perm), _ptr(src), int(width), _ptr(dst), _ptr(workspace), int(ws_bytes),
                               _stream(stream)), "ec2moe_route")


def ec2moe_route_noalloc(desc, topk_idx, counts, offsets, perm, inv_perm=None, src=None, width=0, dst=None,
                         stream=None):
    """ec2moe_route without a workspace: the histograms use a fixed array inside the library."""
    _check(load().ec2moe_route_noalloc(_dref(desc), _ptr(topk_idx), _ptr(counts), _ptr(offsets), _ptr(perm),
                                       _ptr(inv_perm), _ptr(src), int(width), _ptr(dst), _stream(stream)),
           "ec2moe_route_noalloc")


def ec2moe_experts(desc, X_perm, offsets, W1, W3, W2, topk_w, perm, slot_out, workspace, ws_bytes, stream=None):
    _check(load().ec2moe_experts(_dref(desc), _ptr(X_perm), _ptr(offsets), _ptr(W1), _ptr(W3), _ptr(W2),
                                 _ptr(topk_w), _ptr(perm), _ptr(slot_out), _ptr(workspace), int(ws_bytes),
                                 _stream(stream)), "ec2moe_experts")


def ec2moe_shared_experts(desc, X, W1s, W3s, W2s, shared_out, workspace, ws_bytes, stream=None):
    _check(load().ec2moe_shared_experts(_dref(desc), _ptr(X), _ptr(W1s), _ptr(W3s), _ptr(W2s),
                                        _ptr(shared_out), _ptr(workspace), int(ws_bytes), _stream(stream)),
           "ec2moe_shared_experts")


def ec2moe_combine(desc, slot_out, shared_out, Y, stream=None):
    _check(load().ec2moe_combine(_dref(desc), _ptr(slot_out), _ptr(shared_out), _ptr(Y), _stream(stream)),
           "ec2moe_combine")


def ec2moe_lr_encode(desc, X, V_enc, Z, stream=None):
    _check(load().ec2moe_lr_encode(_dref(desc), _ptr(X), _ptr(V_enc), _ptr(Z), _stream(stream)),
           "ec2moe_lr_encode")


def ec2moe_lr_decode(desc, Z, V_dec, X_hat, stream=None):
    _check(load().ec2moe_lr_decode(_dref(desc), _ptr(Z), _ptr(V_dec), _ptr(X_hat), _stream(stream)),
           "ec2moe_lr_decode")


def ec2moe_layer_forward(desc, weights: LayerWeights, X, mask, Y, topk_idx, topk_w, counts, Z, workspace, ws_bytes,
                         stream=None):
    _check(load().ec2moe_layer_forward(_dref(desc), ctypes.byref(weights), _ptr(X), _mask(mask), _ptr(Y),
                                       _ptr(topk_idx), _ptr(topk_w), _ptr(counts), _ptr(Z), _ptr(workspace),
                                       int(ws_bytes), _stream(stream)), "ec2moe_layer_forward")


def ec2moe_pipelined_workspace_size(desc: LayerDesc, n_micro: int) -> int:
    return int(load().ec2moe_pipelined_workspace_size(_dref(desc), int(n_micro)))


def ec2moe_layer_forward_pipelined(desc, weights: LayerWeights, X, mask, Y, topk_idx, topk_w, counts, Z, workspace,
                                   ws_bytes, n_micro, stream_end=None, stream_cloud=None):
    _check(load().ec2moe_layer_forward_pipelined(_dref(desc), ctypes.byref(weights), _ptr(X), _mask(mask), _ptr(Y),
                                                 _ptr(topk_idx), _ptr(topk_w), _ptr(counts), _ptr(Z),
                                                 _ptr(workspace), int(ws_bytes), int(n_micro), _stream(stream_end),
                                                 _stream(stream_cloud)), "ec2moe_layer_forward_pipelined")


def ec2moe_last_device_error(stream=None) -> int:
    return int(load().ec2moe_last_device_error(_stream(stream)))


def ec2moe_last_launch_count() -> int:
    return int(load().ec2moe_last_launch_count())


def ec2moe_profile_enable(enable: bool = True) -> None:
    _check(load().ec2moe_profile_enable(1 if enable else 0), "ec2moe_profile_enable")


def ec2moe_profile_only(launch_index: int) -> None:
    """Bracket only the launch_index-th launch of each later call (-1: every launch)."""
    _check(load().ec2moe_profile_only(int(launch_index)), "ec2moe_profile_only")


def ec2moe_profile_count() -> int:
    return int(load().ec2moe_profile_count())


def ec2moe_profile_read(i: int):
    """(name, milliseconds) of the i-th recorded launch."""
    name = ctypes.c_char_p()
    ms = ctypes.c_float()
    _check(load().ec2moe_profile_read(int(i), ctypes.byref(name), ctypes.byref(ms)), "ec2moe_profile_read")
    return name.value.decode(), float(ms.value)


def ec2moe_profile_reset() -> None:
    load().ec2moe_profile_reset()


def ec2moe_set_wait_budget(cycles: int) -> None:
    _check(load().ec2moe_set_wait_budget(int(cycles)), "ec2moe_set_wait_budget")


def ec2moe_get_wait_budget() -> int:
    return int(load().ec2moe_get_wait_budget())


# ----------------------------------------------------------------- scheduler (host)
def _dbl_array(values):
    vals = [float(v) for v in values]
    return (ctypes.c_double * max(1, len(vals)))(*vals), len(vals)


def ec2moe_schedule(cost, comm, load_end=0.0, load_cloud=0.0, T_end=float("inf"), beta=0.0, eps=1e-9):
    """Eq. 10-11 placement.  Returns (location list of END/CLOUD, visit order,
    final End load, final Cloud load)."""
    c, n = _dbl_array(cost)
    m, n2 = _dbl_array(comm)
    if n != n2:
        raise ValueError("cost and comm differ in length")
    loc = (ctypes.c_int32 * max(1, n))()
    order = (ctypes.c_int32 * max(1, n))()
    le, lc = ctypes.c_double(), ctypes.c_double()
    _check(load().ec2moe_schedule(n, ctypes.addressof(c), ctypes.addressof(m), float(load_end), float(load_cloud),
                                  float(T_end), float(beta), float(eps), ctypes.addressof(loc),
                                  ctypes.addressof(order), ctypes.addressof(le), ctypes.addressof(lc)),
           "ec2moe_schedule")
    return list(loc)[:n], list(order)[:n], le.value, lc.value


def ec2moe_schedule_objective(cost, comm, location, rate_end, rate_cloud, alpha) -> float:
    """Eq. 9 objective of a placement."""
    c, n = _dbl_array(cost)
    m, _ = _dbl_array(comm)
    loc = (ctypes.c_int32 * max(1, n))(*[int(v) for v in location])
    out = ctypes.c_double()
    _check(load().ec2moe_schedule_objective(n, ctypes.addressof(c), ctypes.addressof(m), ctypes.addressof(loc),
                                            float(rate_end), float(rate_cloud), float(alpha),
                                            ctypes.addressof(out)), "ec2moe_schedule_objective")
    return out.value


def ec2moe_expert_tasks(desc, counts):
    """Route-aware tasks from a host histogram: (expert ids, costs, comms)."""
    E = int(desc.E)
    cnt = (ctypes.c_int32 * E)(*[int(v) for v in counts])
    ids = (ctypes.c_int32 * E)()
    cost = (ctypes.c_double * E)()
    comm = (ctypes.c_double * E)()
    nt = ctypes.c_int32()
    _check(load().ec2moe_expert_tasks(_dref(desc), ctypes.addressof(cnt), ctypes.addressof(ids),
                                      ctypes.addressof(cost), ctypes.addressof(comm), ctypes.addressof(nt)),
           "ec2moe_expert_tasks")
    n = nt.value
    return list(ids)[:n], list(cost)[:n], list(comm)[:n]
