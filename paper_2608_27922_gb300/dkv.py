"""Thin ctypes binding of libdkv.so (include/dkv.h), with the same names as the C ABI.

Only argument marshalling happens here: torch tensors are checked for device,
dtype, shape and contiguity and passed as raw device pointers; every step of
the bank update and of attention runs in the CUDA library.  There is no CPU or
PyTorch fallback: if the library cannot be loaded, ``lib()`` raises.

``BankLayer`` is a convenience owner of one layer's caller-owned buffers
(bank tensors and workspace, allocated with torch) around a ``dkv_bank_t``.
"""
from __future__ import annotations

import ctypes
import os
from typing import Dict, List, Optional, Sequence, Tuple

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "lib", "libdkv.so")

DKV_OK = 0
DKV_DTYPE_BF16, DKV_DTYPE_FP32 = 0, 1
DKV_SCORE_TENSOR, DKV_SCORE_FP32 = 0, 1
DKV_ORDER_SCORE, DKV_ORDER_SOURCE = 0, 1
DKV_DESC_K, DKV_DESC_KV = 0, 1
DKV_EVICT_MANDATORY_DENSEST, DKV_EVICT_DENSEST, DKV_EVICT_MANDATORY_SOURCE = 0, 1, 2
STATUS = {0: "DKV_OK", 1: "DKV_ERR_ARG", 2: "DKV_ERR_SHAPE", 3: "DKV_ERR_STATE", 4: "DKV_ERR_CUDA",
          5: "DKV_ERR_NOMEM", 6: "DKV_ERR_TIMEOUT", 7: "DKV_ERR_UNSUPPORTED", 8: "DKV_ERR_DEVICE"}


class dkv_params_t(ctypes.Structure):
    _fields_ = [("tau", ctypes.c_float), ("sigma", ctypes.c_float), ("p", ctypes.c_float),
                ("eps", ctypes.c_float), ("delta", ctypes.c_float), ("sync_heads", ctypes.c_int32),
                ("score_mode", ctypes.c_int32), ("order", ctypes.c_int32), ("eviction", ctypes.c_int32),
                ("refresh_baselines", ctypes.c_int32), ("layer_heads", ctypes.c_int32),
                ("descriptor", ctypes.c_int32)]


class dkv_buffers_t(ctypes.Structure):
    _fields_ = [("k", ctypes.c_void_p), ("v", ctypes.c_void_p), ("rho", ctypes.c_void_p),
                ("base", ctypes.c_void_p), ("knorm", ctypes.c_void_p), ("prov_step", ctypes.c_void_p),
                ("prov_src", ctypes.c_void_p), ("occupancy", ctypes.c_void_p),
                ("workspace", ctypes.c_void_p), ("workspace_bytes", ctypes.c_size_t)]


class dkv_layer_stats_t(ctypes.Structure):
    _fields_ = [("r_star", ctypes.c_int32), ("rmax", ctypes.c_int32), ("n_candidates", ctypes.c_int32),
                ("empty_init", ctypes.c_int32)]


class dkv_head_stats_t(ctypes.Structure):
    _fields_ = [("occupancy_before", ctypes.c_int32), ("occupancy_after", ctypes.c_int32),
                ("admitted", ctypes.c_int32), ("evicted", ctypes.c_int32), ("mandatory", ctypes.c_int32),
                ("pre_violators", ctypes.c_int32)]


class dkv_intermediates_t(ctypes.Structure):
    _fields_ = [("score", ctypes.c_void_p), ("perm", ctypes.c_void_p), ("cross", ctypes.c_void_p),
                ("rho_tilde", ctypes.c_void_p), ("slot_new", ctypes.c_void_p), ("n_max", ctypes.c_int64),
                ("M_max", ctypes.c_int64)]


# (name, restype, argtypes) of every exported symbol declared in include/dkv.h
_P = ctypes.c_void_p
_I = ctypes.c_int32
SIGNATURES = [
    ("dkv_status_str", ctypes.c_char_p, [_I]),
    ("dkv_version", _I, []),
    ("dkv_params_default", _I, [ctypes.POINTER(dkv_params_t), _I]),
    ("dkv_bank_workspace_size", ctypes.c_size_t, [_I, _I, ctypes.POINTER(ctypes.c_int32), _I, _I]),
    ("dkv_bank_workspace_size_ex", ctypes.c_size_t, [_I, _I, ctypes.POINTER(ctypes.c_int32), _I, _I,
                                                     ctypes.POINTER(dkv_params_t)]),
    ("dkv_bank_create", _I, [ctypes.POINTER(_P), _I, _I, ctypes.POINTER(ctypes.c_int32), _I, _I,
                             ctypes.POINTER(dkv_params_t), ctypes.POINTER(dkv_buffers_t)]),
    ("dkv_bank_destroy", None, [_P]),
    ("dkv_bank_reset", _I, [_P, _P]),
    ("dkv_bank_admit", _I, [_P, _P, _P, _I, ctypes.c_int64, _P]),
    ("dkv_bank_admit_rope", _I, [_P, _P, _P, _I, ctypes.c_int64, _P, _P, _I, _P]),
    ("dkv_bank_compress", _I, [_P, _P]),
    ("dkv_bank_evict", _I, [_P, _P]),
    ("dkv_bank_commit", _I, [_P, _P]),
    ("dkv_bank_attend", _I, [_P, _P, _I, _P, _P, _I, _P, _P]),
    ("dkv_bank_import", _I, [_P, ctypes.POINTER(ctypes.c_int32), _P]),
    ("dkv_bank_export", _I, [_P, ctypes.POINTER(dkv_buffers_t)]),
    ("dkv_bank_sync", _I, [_P]),
    ("dkv_bank_stats", _I, [_P, ctypes.POINTER(dkv_layer_stats_t), ctypes.POINTER(dkv_head_stats_t)]),
    ("dkv_bank_occupancy", _I, [_P, ctypes.POINTER(ctypes.c_int32)]),
    ("dkv_bank_intermediates", _I, [_P, ctypes.POINTER(dkv_intermediates_t)]),
    ("dkv_bank_set_timing", _I, [_P, _I]),
    ("dkv_bank_kernel_times", _I, [_P, _I, ctypes.c_char_p, ctypes.POINTER(ctypes.c_int32),
                                   ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_int32)]),
    ("dkv_candidate_order_noalloc", _I, [_P, _P, _I, _P, _I, _I, _I, ctypes.POINTER(dkv_params_t), _P, _P, _P]),
    ("dkv_selftest_wait_timeout", _I, [_I, ctypes.POINTER(ctypes.c_int64)]),
    ("dkv_sequential_scratch_size", ctypes.c_size_t, [_I, _I, _I, _I]),
    ("dkv_bank_update_sequential", _I, [_P, _P, _P, _I, ctypes.c_int64, _P, ctypes.c_size_t, _P]),
]

DKV_NOALLOC_MAX_N = 16384

_LIB: Optional[ctypes.CDLL] = None


def lib() -> ctypes.CDLL:
    """Loads libdkv.so (built in-tree by ``build.py``); raises if it is missing."""
    global _LIB
    if _LIB is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with paper_2608_27922_gb300.build.build()")
        L = ctypes.CDLL(LIB_PATH)
        for name, res, args in SIGNATURES:
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _LIB = L
    return _LIB


class DkvError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {STATUS.get(status, status)} ({lib().dkv_status_str(status).decode()})")


def _check(status: int, what: str) -> None:
    if status != DKV_OK:
        raise DkvError(status, what)


def _stream(stream) -> int:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


def _ptr(t) -> int:
    if t is None:
        return 0
    if isinstance(t, int):
        return t
    if not t.is_cuda or not t.is_contiguous():
        raise ValueError("expected a contiguous CUDA tensor")
    return t.data_ptr()


def _i32(xs: Sequence[int]):
    return (ctypes.c_int32 * len(xs))(*[int(x) for x in xs])


# ----------------------------------------------------------------- C ABI, same names
def dkv_version() -> int:
    return lib().dkv_version()


def dkv_params_default(d: int) -> dkv_params_t:
    p = dkv_params_t()
    _check(lib().dkv_params_default(ctypes.byref(p), d), "dkv_params_default")
    return p


def dkv_bank_workspace_size(H: int, d: int, budgets: Sequence[int], n_max: int, dtype: int,
                            params: Optional[dkv_params_t] = None) -> int:
    if params is None:
        return int(lib().dkv_bank_workspace_size(H, d, _i32(budgets), n_max, dtype))
    return int(lib().dkv_bank_workspace_size_ex(H, d, _i32(budgets), n_max, dtype, ctypes.byref(params)))


def dkv_bank_create(H: int, d: int, budgets: Sequence[int], n_max: int, dtype: int, params: dkv_params_t,
                    buffers: dkv_buffers_t) -> int:
    h = ctypes.c_void_p()
    _check(lib().dkv_bank_create(ctypes.byref(h), H, d, _i32(budgets), n_max, dtype, ctypes.byref(params),
                                 ctypes.byref(buffers)), "dkv_bank_create")
    return h.value


def dkv_bank_destroy(bank: int) -> None:
    lib().dkv_bank_destroy(bank)


def dkv_bank_reset(bank: int, stream=None) -> None:
    _check(lib().dkv_bank_reset(bank, _stream(stream)), "dkv_bank_reset")


def dkv_bank_admit(bank: int, Kc, Vc, N: int, step: int, stream=None) -> None:
    _check(lib().dkv_bank_admit(bank, _ptr(Kc), _ptr(Vc), N, step, _stream(stream)), "dkv_bank_admit")


DKV_ROPE_INTERLEAVED, DKV_ROPE_HALF = 0, 1


def dkv_bank_admit_rope(bank: int, Kc, Vc, N: int, step: int, t_coord, theta, layout: int, stream=None) -> None:
    _check(lib().dkv_bank_admit_rope(bank, _ptr(Kc), _ptr(Vc), N, step, _ptr(t_coord), _ptr(theta), layout,
                                     _stream(stream)), "dkv_bank_admit_rope")


def dkv_sequential_scratch_size(H: int, d: int, n_max: int, dtype: int) -> int:
    return int(lib().dkv_sequential_scratch_size(H, d, n_max, dtype))


def dkv_bank_update_sequential(bank: int, Kc, Vc, N: int, step: int, scratch, scratch_bytes: int,
                               stream=None) -> None:
    _check(lib().dkv_bank_update_sequential(bank, _ptr(Kc), _ptr(Vc), N, step, _ptr(scratch), scratch_bytes,
                                            _stream(stream)), "dkv_bank_update_sequential")


def dkv_bank_compress(bank: int, stream=None) -> None:
    _check(lib().dkv_bank_compress(bank, _stream(stream)), "dkv_bank_compress")


def dkv_bank_evict(bank: int, stream=None) -> None:
    _check(lib().dkv_bank_evict(bank, _stream(stream)), "dkv_bank_evict")


def dkv_bank_commit(bank: int, stream=None) -> None:
    _check(lib().dkv_bank_commit(bank, _stream(stream)), "dkv_bank_commit")


def dkv_bank_attend(bank: int, Q, Nq: int, Kw, Vw, W: int, O, stream=None) -> None:
    _check(lib().dkv_bank_attend(bank, _ptr(Q), Nq, _ptr(Kw), _ptr(Vw), W, _ptr(O), _stream(stream)),
           "dkv_bank_attend")


def dkv_bank_import(bank: int, occupancy: Sequence[int], stream=None) -> None:
    _check(lib().dkv_bank_import(bank, _i32(occupancy), _stream(stream)), "dkv_bank_import")


def dkv_bank_export(bank: int, dst: dkv_buffers_t) -> None:
    _check(lib().dkv_bank_export(bank, ctypes.byref(dst)), "dkv_bank_export")


def dkv_bank_sync(bank: int) -> None:
    _check(lib().dkv_bank_sync(bank), "dkv_bank_sync")


def dkv_bank_stats(bank: int, H: int, n_layers: int = 1) -> Tuple[List[dkv_layer_stats_t], List[dkv_head_stats_t]]:
    Ls = (dkv_layer_stats_t * n_layers)()
    arr = (dkv_head_stats_t * H)()
    _check(lib().dkv_bank_stats(bank, Ls, arr), "dkv_bank_stats")
    return list(Ls), list(arr)


def dkv_bank_occupancy(bank: int, H: int) -> List[int]:
    arr = (ctypes.c_int32 * H)()
    _check(lib().dkv_bank_occupancy(bank, arr), "dkv_bank_occupancy")
    return list(arr)


def dkv_bank_intermediates(bank: int) -> dkv_intermediates_t:
    x = dkv_intermediates_t()
    _check(lib().dkv_bank_intermediates(bank, ctypes.byref(x)), "dkv_bank_intermediates")
    return x


def dkv_bank_set_timing(bank: int, enable) -> None:
    """enable: False/0 off, True/1 every kernel, 2 attention launches only (others counted)."""
    _check(lib().dkv_bank_set_timing(bank, int(enable)), "dkv_bank_set_timing")


def dkv_bank_kernel_times(bank: int) -> Dict[str, Tuple[int, float]]:
    n = ctypes.c_int32()
    _check(lib().dkv_bank_kernel_times(bank, 0, None, None, None, ctypes.byref(n)), "dkv_bank_kernel_times")
    k = n.value
    names = ctypes.create_string_buffer(48 * max(k, 1))
    launches = (ctypes.c_int32 * max(k, 1))()
    ms = (ctypes.c_double * max(k, 1))()
    _check(lib().dkv_bank_kernel_times(bank, k, names, launches, ms, ctypes.byref(n)), "dkv_bank_kernel_times")
    out = {}
    for i in range(min(k, n.value)):
        nm = names.raw[48 * i:48 * (i + 1)].split(b"\0", 1)[0].decode()
        out[nm] = (int(launches[i]), float(ms[i]))
    return out


def dkv_candidate_order_noalloc(K_bank, base, m: int, Kc, N: int, d: int, dtype: int, params: dkv_params_t,
                                scores_out, perm_out, stream=None) -> None:
    """Eq. 6 scores and their stable order for one head, with no device allocation
    (for callers that cannot allocate; see include/dkv.h)."""
    _check(lib().dkv_candidate_order_noalloc(_ptr(K_bank) if m > 0 else 0, _ptr(base) if m > 0 else 0, m,
                                             _ptr(Kc), N, d, dtype, ctypes.byref(params), _ptr(scores_out),
                                             _ptr(perm_out), _stream(stream)), "dkv_candidate_order_noalloc")


def dkv_selftest_wait_timeout(limit_us: int):
    """Runs the bounded-wait self-test; returns (status, elapsed_ns).  DKV_ERR_TIMEOUT (6)
    is the expected status: the wait gave up after limit_us as designed."""
    el = ctypes.c_int64(0)
    st = lib().dkv_selftest_wait_timeout(int(limit_us), ctypes.byref(el))
    return int(st), int(el.value)


# ----------------------------------------------------------------- buffer owner
_TORCH_DTYPE = {DKV_DTYPE_BF16: torch.bfloat16, DKV_DTYPE_FP32: torch.float32}


def _view(ptr: int, shape, dtype: torch.dtype, device) -> torch.Tensor:
    """Wraps a device pointer owned by the library handle as a read-only-by-convention tensor."""
    n = 1
    for s in shape:
        n *= s
    esize = torch.empty(0, dtype=dtype).element_size()

    class _Arr:
        __cuda_array_interface__ = {
            "shape": (n,), "typestr": {torch.float32: "<f4", torch.int32: "<i4"}[dtype],
            "data": (ptr, False), "version": 3, "strides": (esize,)}

    return torch.as_tensor(_Arr(), device=device).view(*shape)


class BankLayer:
    """H per-head banks (one layer, or H / layer_heads layers when the layer_heads
    parameter is set): allocates the caller-owned buffers with torch and drives the C
    ABI.  All methods enqueue on the current (or given) stream."""

    def __init__(self, H: int, d: int, budgets: Sequence[int], n_max: int, dtype: torch.dtype = torch.bfloat16,
                 params: Optional[dkv_params_t] = None, device="cuda", **param_overrides):
        self.H, self.d, self.n_max = H, d, n_max
        self.budgets = [int(b) for b in budgets]
        assert len(self.budgets) == H
        self.M_max = max(self.budgets)
        self.dtype_code = {torch.bfloat16: DKV_DTYPE_BF16, torch.float32: DKV_DTYPE_FP32}[dtype]
        self.dtype = dtype
        dev = torch.device(device)
        if dev.type == "cuda" and dev.index is None:
            dev = torch.device("cuda", torch.cuda.current_device())
        self.device = dev
        p = params if params is not None else dkv_params_default(d)
        for k, v in param_overrides.items():
            setattr(p, k, v)
        self.params = p
        self.n_layers = H // p.layer_heads if p.layer_heads > 0 else 1
        dev = self.device
        self.k = torch.zeros(H, self.M_max, d, dtype=dtype, device=dev)
        self.v = torch.zeros(H, self.M_max, d, dtype=dtype, device=dev)
        self.rho = torch.zeros(H, self.M_max, dtype=torch.float32, device=dev)
        self.base = torch.zeros(H, self.M_max, dtype=torch.float32, device=dev)
        self.knorm = torch.zeros(H, self.M_max, dtype=torch.float32, device=dev)
        self.prov_step = torch.full((H, self.M_max), -1, dtype=torch.int64, device=dev)
        self.prov_src = torch.full((H, self.M_max), -1, dtype=torch.int32, device=dev)
        self.occupancy = torch.zeros(H, dtype=torch.int32, device=dev)
        ws = dkv_bank_workspace_size(H, d, self.budgets, n_max, self.dtype_code, p)
        if ws == 0:
            raise ValueError("invalid bank shape")
        self.workspace = torch.empty(ws, dtype=torch.uint8, device=dev)
        bufs = dkv_buffers_t(self.k.data_ptr(), self.v.data_ptr(), self.rho.data_ptr(), self.base.data_ptr(),
                             self.knorm.data_ptr(), self.prov_step.data_ptr(), self.prov_src.data_ptr(),
                             self.occupancy.data_ptr(), self.workspace.data_ptr(), ws)
        self.handle = dkv_bank_create(H, d, self.budgets, n_max, self.dtype_code, p, bufs)

    def close(self):
        if getattr(self, "handle", None):
            dkv_bank_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _chk(self, t: torch.Tensor, shape, name: str):
        if t.dtype != self.dtype or tuple(t.shape) != tuple(shape) or not t.is_contiguous() or t.device != self.device:
            raise ValueError(f"{name}: expected contiguous {self.dtype} {tuple(shape)} on {self.device}, "
                             f"got {t.dtype} {tuple(t.shape)} on {t.device}")

    def reset(self, stream=None):
        dkv_bank_reset(self.handle, stream)

    def admit(self, Kc: torch.Tensor, Vc: torch.Tensor, step: int, stream=None, t_coord=None, theta=None,
              rope_layout: int = DKV_ROPE_INTERLEAVED):
        """Steps 1-2.  With t_coord (int32 [N]) and theta (fp32 [d/2]) on the device, the
        keys are first rotated back to temporal rotary coordinate 0 (dkv_bank_admit_rope)."""
        N = Kc.shape[1]
        self._chk(Kc, (self.H, N, self.d), "Kc")
        self._chk(Vc, (self.H, N, self.d), "Vc")
        if (t_coord is None) != (theta is None):
            raise ValueError("t_coord and theta go together")
        if t_coord is None:
            self._pending = (Kc, Vc)   # keep the candidates alive until commit
            dkv_bank_admit(self.handle, Kc, Vc, N, step, stream)
            return
        for x, dt, shape, name in ((t_coord, torch.int32, (N,), "t_coord"), (theta, torch.float32, (self.d // 2,), "theta")):
            if x.dtype != dt or tuple(x.shape) != shape or not x.is_contiguous() or x.device != self.device:
                raise ValueError(f"{name}: expected contiguous {dt} {shape} on {self.device}")
        self._pending = (Kc, Vc, t_coord, theta)
        dkv_bank_admit_rope(self.handle, Kc, Vc, N, step, t_coord, theta, rope_layout, stream)

    def compress(self, stream=None):
        dkv_bank_compress(self.handle, stream)

    def evict(self, stream=None):
        """First half of compress; leaves k, v and occupancy untouched."""
        dkv_bank_evict(self.handle, stream)

    def commit(self, stream=None):
        """Second half of compress; order every reader of the old bank before it."""
        dkv_bank_commit(self.handle, stream)

    def update(self, Kc: torch.Tensor, Vc: torch.Tensor, step: int, stream=None, **rope):
        self.admit(Kc, Vc, step, stream, **rope)
        self.compress(stream)

    def update_sequential(self, Kc: torch.Tensor, Vc: torch.Tensor, step: int, stream=None):
        """Within-block competition: the block's candidates offered one at a time (the
        C ABI's dkv_bank_update_sequential); synchronises once with the stream."""
        N = Kc.shape[1]
        self._chk(Kc, (self.H, N, self.d), "Kc")
        self._chk(Vc, (self.H, N, self.d), "Vc")
        if getattr(self, "_seq_scratch", None) is None:
            n = dkv_sequential_scratch_size(self.H, self.d, self.n_max, self.dtype_code)
            self._seq_scratch = torch.empty(n, dtype=torch.uint8, device=self.device)
        dkv_bank_update_sequential(self.handle, Kc, Vc, N, step, self._seq_scratch, self._seq_scratch.numel(),
                                   stream)

    def attend(self, Q: torch.Tensor, Kw: Optional[torch.Tensor], Vw: Optional[torch.Tensor],
               out: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
        Nq = Q.shape[1]
        self._chk(Q, (self.H, Nq, self.d), "Q")
        W = 0 if Kw is None else Kw.shape[1]
        if W:
            self._chk(Kw, (self.H, W, self.d), "Kw")
            self._chk(Vw, (self.H, W, self.d), "Vw")
        if out is None:
            out = torch.empty_like(Q)
        self._chk(out, (self.H, Nq, self.d), "out")
        dkv_bank_attend(self.handle, Q, Nq, Kw if W else None, Vw if W else None, W, out, stream)
        return out

    def import_state(self, occupancy: Sequence[int], stream=None):
        dkv_bank_import(self.handle, occupancy, stream)

    def export_state(self, device="cpu") -> Dict[str, torch.Tensor]:
        """Checkpoint of every head (k, v, rho, base, prov_step, prov_src, occupancy), copied
        by dkv_bank_export into new tensors on `device` (host tensors are pinned)."""
        dev = torch.device(device)
        pin = dev.type == "cpu"
        H, M, d = self.H, self.M_max, self.d

        def new(shape, dtype):
            return torch.empty(shape, dtype=dtype, device=dev, pin_memory=pin)
        out = {"k": new((H, M, d), self.dtype), "v": new((H, M, d), self.dtype),
               "rho": new((H, M), torch.float32), "base": new((H, M), torch.float32),
               "prov_step": new((H, M), torch.int64), "prov_src": new((H, M), torch.int32),
               "occupancy": new((H,), torch.int32)}
        dst = dkv_buffers_t()
        for name in ("k", "v", "rho", "base", "prov_step", "prov_src", "occupancy"):
            setattr(dst, name, out[name].data_ptr())
        dkv_bank_export(self.handle, dst)
        return out

    def sync(self):
        dkv_bank_sync(self.handle)

    def stats(self):
        """(statistics of the first layer, per-head statistics of every head)."""
        Ls, hs = dkv_bank_stats(self.handle, self.H, self.n_layers)
        return Ls[0], hs

    def layer_stats(self) -> List[dkv_layer_stats_t]:
        """Statistics of each of the handle's layers (params.layer_heads heads each)."""
        return dkv_bank_stats(self.handle, self.H, self.n_layers)[0]

    def occupancy_host(self) -> List[int]:
        return dkv_bank_occupancy(self.handle, self.H)

    def intermediates(self) -> Dict[str, torch.Tensor]:
        x = dkv_bank_intermediates(self.handle)
        H, n, M = self.H, int(x.n_max), int(x.M_max)
        return {"score": _view(x.score, (H, n), torch.float32, self.device),
                "perm": _view(x.perm, (H, n), torch.int32, self.device),
                "cross": _view(x.cross, (H, M), torch.int32, self.device),
                "rho_tilde": _view(x.rho_tilde, (H, M), torch.float32, self.device),
                "slot_new": _view(x.slot_new, (H, n), torch.int32, self.device)}

    def set_timing(self, on: bool, attention_only: bool = False):
        dkv_bank_set_timing(self.handle, 2 if (on and attention_only) else int(bool(on)))

    def kernel_times(self):
        return dkv_bank_kernel_times(self.handle)
