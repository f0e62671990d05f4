"""dMoE block-routed MoE-layer forward on GB300 (sm_103a): Python binding of libdmoe.so.

The functions below carry the names of the C ABI in ``include/dmoe.h`` and only marshal
arguments: torch tensors (CUDA, contiguous, of the documented dtype) become device
pointers, ``None`` becomes NULL, and the current torch CUDA stream is used unless one is
given. Every step of the forward runs in the library's CUDA kernels; there is no other
implementation in this package, and importing it fails when the library is not built.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Tuple

import torch

__all__ = [
    "DMOE_ROUTE_TOKEN", "DMOE_ROUTE_BLOCK", "DmoeError", "LayerDesc", "make_desc",
    "dmoe_workspace_size", "dmoe_router", "dmoe_dispatch", "dmoe_moe_forward",
    "dmoe_layer_forward", "dmoe_get_device_error", "dmoe_status_string", "dmoe_abi_version",
    "dmoe_layer_forward_launches",
    "alloc_workspace", "LIB_PATH", "dmoe_set_profile_events", "KERNELS",
]

DMOE_ROUTE_TOKEN = 0
DMOE_ROUTE_BLOCK = 1

DMOE_OK = 0
STATUS_NAMES = {0: "DMOE_OK", 1: "DMOE_ERR_INVALID_ARG", 2: "DMOE_ERR_UNSUPPORTED",
                3: "DMOE_ERR_WORKSPACE", 4: "DMOE_ERR_CUDA", 5: "DMOE_ERR_DEVICE",
                6: "DMOE_ERR_TIMEOUT"}

# DMOE_LIB selects another build of the same library (for example one compiled with other
# flags); by default the in-tree libdmoe.so
LIB_PATH = os.environ.get("DMOE_LIB") or os.path.join(
    os.path.dirname(os.path.abspath(__file__)), "libdmoe.so")


class LayerDesc(ctypes.Structure):
    """dmoe_layer_desc (include/dmoe.h)."""
    _fields_ = [("d_model", ctypes.c_int32), ("n_experts", ctypes.c_int32),
                ("top_k", ctypes.c_int32), ("d_ff", ctypes.c_int32),
                ("d_ff_shared", ctypes.c_int32), ("block_size", ctypes.c_int32),
                ("n_blocks", ctypes.c_int32), ("mode", ctypes.c_int32),
                ("top_p", ctypes.c_float), ("block_top_k", ctypes.c_int32)]

    @property
    def T(self) -> int:
        return self.n_blocks * self.block_size


def make_desc(d_model, n_experts, top_k, d_ff, d_ff_shared, block_size, n_blocks,
              mode=DMOE_ROUTE_BLOCK, top_p=0.0, block_top_k=0) -> LayerDesc:
    return LayerDesc(d_model, n_experts, top_k, d_ff, d_ff_shared, block_size, n_blocks,
                     mode, float(top_p), int(block_top_k))


class DmoeError(RuntimeError):
    def __init__(self, status: int, where: str, detail: str = ""):
        self.status = status
        msg = f"{where}: {STATUS_NAMES.get(status, status)}"
        if detail:
            msg += f" ({detail})"
        super().__init__(msg)


def _load() -> ctypes.CDLL:
    if not os.path.exists(LIB_PATH):
        raise ImportError(
            f"{LIB_PATH} is not built; run `python -c 'import __graft_entry__ as g; g.build()'`")
    lib = ctypes.CDLL(LIB_PATH)
    P = ctypes.c_void_p
    D = ctypes.POINTER(LayerDesc)
    st = ctypes.c_int
    lib.dmoe_workspace_size.argtypes = [D, ctypes.POINTER(ctypes.c_size_t)]
    lib.dmoe_workspace_size.restype = st
    lib.dmoe_router.argtypes = [D, P, P, P, P, P, P, P, P, P, ctypes.c_size_t, P]
    lib.dmoe_router.restype = st
    lib.dmoe_router_prepare.argtypes = [D, P, P, ctypes.c_size_t, P]
    lib.dmoe_router_prepare.restype = st
    lib.dmoe_dispatch.argtypes = [D, P, P, P, P, P, P, P, ctypes.c_size_t, P]
    lib.dmoe_dispatch.restype = st
    lib.dmoe_moe_forward.argtypes = [D] + [P] * 14 + [P, ctypes.c_size_t, P]
    lib.dmoe_moe_forward.restype = st
    lib.dmoe_layer_forward.argtypes = [D] + [P] * 14 + [P, ctypes.c_size_t, P]
    lib.dmoe_layer_forward.restype = st
    lib.dmoe_get_device_error.argtypes = [P, P, ctypes.POINTER(ctypes.c_int32)]
    lib.dmoe_get_device_error.restype = st
    lib.dmoe_status_string.argtypes = [ctypes.c_int]
    lib.dmoe_status_string.restype = ctypes.c_char_p
    lib.dmoe_last_error_message.argtypes = []
    lib.dmoe_last_error_message.restype = ctypes.c_char_p
    lib.dmoe_abi_version.argtypes = []
    lib.dmoe_abi_version.restype = ctypes.c_int32
    lib.dmoe_layer_forward_launches.argtypes = [ctypes.POINTER(LayerDesc)]
    lib.dmoe_layer_forward_launches.restype = ctypes.c_int32
    lib.dmoe_set_profile_events.argtypes = [ctypes.c_int32, P, P]
    lib.dmoe_set_profile_events.restype = st
    lib.dmoe_set_debug_hold.argtypes = [P, ctypes.c_int32, P]
    lib.dmoe_set_debug_hold.restype = st
    lib.dmoe_router_no_alloc.argtypes = [D, P, P, P, P, P, P, P, P, P]
    lib.dmoe_router_no_alloc.restype = st
    lib.dmoe_router_no_alloc_device_error.argtypes = [P, ctypes.POINTER(ctypes.c_int32)]
    lib.dmoe_router_no_alloc_device_error.restype = st
    lib.dmoe_no_alloc_scratch.argtypes = [ctypes.POINTER(P), ctypes.POINTER(ctypes.c_size_t)]
    lib.dmoe_no_alloc_scratch.restype = st
    return lib


_lib = _load()


def _check(status: int, where: str) -> None:
    if status != DMOE_OK:
        detail = _lib.dmoe_last_error_message().decode() if status == 4 else ""
        raise DmoeError(status, where, detail)


def _ptr(t, dtype=None, name="tensor"):
    """Device pointer of a contiguous CUDA tensor (None -> NULL; an int is passed through)."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name}: expected a torch.Tensor")
    if not t.is_cuda:
        raise ValueError(f"{name}: must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name}: must be contiguous")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name}: expected {dtype}, got {t.dtype}")
    return t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


def _ws(workspace: torch.Tensor) -> Tuple[int, int]:
    if workspace is None:
        raise ValueError("workspace is required (see alloc_workspace)")
    return _ptr(workspace, torch.uint8, "workspace"), workspace.numel()


def dmoe_workspace_size(desc: LayerDesc) -> int:
    n = ctypes.c_size_t(0)
    _check(_lib.dmoe_workspace_size(ctypes.byref(desc), ctypes.byref(n)), "dmoe_workspace_size")
    return n.value


def alloc_workspace(desc: LayerDesc, device="cuda") -> torch.Tensor:
    """A zeroed uint8 device buffer of dmoe_workspace_size(desc) bytes (torch allocates)."""
    return torch.zeros(dmoe_workspace_size(desc), dtype=torch.uint8, device=device)


def dmoe_router(desc, x, w_r, bias, topk_idx, topk_gate, coreset=None, coreset_size=None,
                probs=None, workspace=None, stream=None) -> None:
    ws, nb = _ws(workspace)
    _check(_lib.dmoe_router(ctypes.byref(desc), _ptr(x, torch.bfloat16, "x"),
                            _ptr(w_r, torch.float32, "w_r"), _ptr(bias, torch.float32, "bias"),
                            _ptr(topk_idx, torch.int32, "topk_idx"),
                            _ptr(topk_gate, torch.float32, "topk_gate"),
                            _ptr(coreset, torch.int32, "coreset"),
                            _ptr(coreset_size, torch.int32, "coreset_size"),
                            _ptr(probs, torch.float32, "probs"), ws, nb, _stream(stream)),
           "dmoe_router")


def dmoe_router_prepare(desc, w_r, workspace, stream=None) -> None:
    ws, nb = _ws(workspace)
    _check(_lib.dmoe_router_prepare(ctypes.byref(desc), _ptr(w_r, torch.float32, "w_r"), ws, nb,
                                    _stream(stream)), "dmoe_router_prepare")


def dmoe_dispatch(desc, topk_idx, n_unique, unique_ids, offsets, rows, pos, workspace=None,
                  stream=None) -> None:
    ws, nb = _ws(workspace)
    i32 = torch.int32
    _check(_lib.dmoe_dispatch(ctypes.byref(desc), _ptr(topk_idx, i32, "topk_idx"),
                              _ptr(n_unique, i32, "n_unique"), _ptr(unique_ids, i32, "unique_ids"),
                              _ptr(offsets, i32, "offsets"), _ptr(rows, i32, "rows"),
                              _ptr(pos, i32, "pos"), ws, nb, _stream(stream)), "dmoe_dispatch")


def dmoe_moe_forward(desc, x, w_gate, w_up, w_down, ws_gate, ws_up, ws_down, topk_gate,
                     n_unique, unique_ids, offsets, rows, pos, y, workspace=None,
                     stream=None) -> None:
    ws, nb = _ws(workspace)
    b, i32 = torch.bfloat16, torch.int32
    _check(_lib.dmoe_moe_forward(
        ctypes.byref(desc), _ptr(x, b, "x"), _ptr(w_gate, b, "w_gate"), _ptr(w_up, b, "w_up"),
        _ptr(w_down, b, "w_down"), _ptr(ws_gate, b, "ws_gate"), _ptr(ws_up, b, "ws_up"),
        _ptr(ws_down, b, "ws_down"), _ptr(topk_gate, torch.float32, "topk_gate"),
        _ptr(n_unique, i32, "n_unique"), _ptr(unique_ids, i32, "unique_ids"),
        _ptr(offsets, i32, "offsets"), _ptr(rows, i32, "rows"), _ptr(pos, i32, "pos"),
        _ptr(y, b, "y"), ws, nb, _stream(stream)), "dmoe_moe_forward")


def dmoe_layer_forward(desc, x, w_r, bias, w_gate, w_up, w_down, ws_gate, ws_up, ws_down, y,
                       topk_idx=None, topk_gate=None, n_unique=None, unique_ids=None,
                       workspace=None, stream=None) -> None:
    ws, nb = _ws(workspace)
    b, i32 = torch.bfloat16, torch.int32
    _check(_lib.dmoe_layer_forward(
        ctypes.byref(desc), _ptr(x, b, "x"), _ptr(w_r, torch.float32, "w_r"),
        _ptr(bias, torch.float32, "bias"), _ptr(w_gate, b, "w_gate"), _ptr(w_up, b, "w_up"),
        _ptr(w_down, b, "w_down"), _ptr(ws_gate, b, "ws_gate"), _ptr(ws_up, b, "ws_up"),
        _ptr(ws_down, b, "ws_down"), _ptr(y, b, "y"), _ptr(topk_idx, i32, "topk_idx"),
        _ptr(topk_gate, torch.float32, "topk_gate"), _ptr(n_unique, i32, "n_unique"),
        _ptr(unique_ids, i32, "unique_ids"), ws, nb, _stream(stream)), "dmoe_layer_forward")


def dmoe_get_device_error(workspace, stream=None) -> Tuple[int, Tuple[int, int, int]]:
    """Synchronises the stream; returns (status, (code, where, value)) and clears the record."""
    info = (ctypes.c_int32 * 4)()
    st = _lib.dmoe_get_device_error(_ptr(workspace, torch.uint8, "workspace"), _stream(stream),
                                    info)
    return st, (info[0], info[1], info[2])


def dmoe_router_no_alloc(desc, x, w_r, bias, topk_idx, topk_gate, coreset=None,
                         coreset_size=None, probs=None, stream=None) -> None:
    """dmoe_router without a workspace (the library's static scratch array)."""
    _check(_lib.dmoe_router_no_alloc(
        ctypes.byref(desc), _ptr(x, torch.bfloat16, "x"), _ptr(w_r, torch.float32, "w_r"),
        _ptr(bias, torch.float32, "bias"), _ptr(topk_idx, torch.int32, "topk_idx"),
        _ptr(topk_gate, torch.float32, "topk_gate"), _ptr(coreset, torch.int32, "coreset"),
        _ptr(coreset_size, torch.int32, "coreset_size"), _ptr(probs, torch.float32, "probs"),
        _stream(stream)), "dmoe_router_no_alloc")


def dmoe_router_no_alloc_device_error(stream=None) -> Tuple[int, Tuple[int, int, int]]:
    """Synchronises the stream; returns (status, (code, where, value)) of the static scratch
    array's fault record and clears it."""
    info = (ctypes.c_int32 * 4)()
    st = _lib.dmoe_router_no_alloc_device_error(_stream(stream), info)
    return st, (info[0], info[1], info[2])


def dmoe_no_alloc_scratch() -> Tuple[int, int]:
    """(device address, bytes) of the static scratch array on the current device."""
    ptr, n = ctypes.c_void_p(0), ctypes.c_size_t(0)
    _check(_lib.dmoe_no_alloc_scratch(ctypes.byref(ptr), ctypes.byref(n)),
           "dmoe_no_alloc_scratch")
    return int(ptr.value or 0), n.value


def dmoe_set_debug_hold(workspace, hold: int, stream=None) -> None:
    """Diagnostic: makes the decode-size expert launch's bounded waits run out while
    `hold` is nonzero (see include/dmoe.h); cleared by dmoe_get_device_error."""
    _check(_lib.dmoe_set_debug_hold(_ptr(workspace, torch.uint8, "workspace"), int(hold),
                                    _stream(stream)), "dmoe_set_debug_hold")


KERNELS = {"router": 0, "dispatch": 1, "gather": 2, "experts": 3, "combine": 4}


def dmoe_set_profile_events(kernel, ev_begin=None, ev_end=None) -> None:
    """Record torch.cuda.Event pairs around every launch of `kernel` (name or id) made by
    later calls on this thread; (None, None) clears."""
    kid = KERNELS[kernel] if isinstance(kernel, str) else int(kernel)
    b = ev_begin.cuda_event if ev_begin is not None else None
    e = ev_end.cuda_event if ev_end is not None else None
    _check(_lib.dmoe_set_profile_events(kid, b, e), "dmoe_set_profile_events")


def dmoe_status_string(status: int) -> str:
    return _lib.dmoe_status_string(status).decode()


def dmoe_abi_version() -> int:
    return _lib.dmoe_abi_version()


def dmoe_layer_forward_launches(desc) -> int:
    """Kernel launches of one dmoe_layer_forward call for `desc` (-1: invalid desc)."""
    return _lib.dmoe_layer_forward_launches(ctypes.byref(desc))
