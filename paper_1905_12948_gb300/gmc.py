"""Python binding of libgmc (include/gmc.h): argument marshalling only.

The functions ``gmc_*`` below carry the C ABI names and arguments one to one;
``GMC`` wraps a handle for torch tensors. Every step of the method runs in the
library's CUDA kernels: there is no CPU path here, and loading fails loudly
when the library has not been built.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Tuple

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libgmc.so")

(GMC_OK, GMC_EINVAL, GMC_ENOMEM, GMC_ECUDA, GMC_ENONFINITE, GMC_ESTATE, GMC_EINTERNAL, GMC_ETOOBIG,
 GMC_ETIMEOUT) = range(9)
GMC_TOPK, GMC_RBGS, GMC_TOPK_APPROX = 0, 1, 2
# Alg. 1, Alg. 3, Alg. 4, and the local-momentum baseline without / with masking
VARIANTS = {"gmc": 0, "server_momentum": 1, "lr_in_residual": 2, "local_momentum": 3,
            "local_momentum_mfm": 4}
GMC_SELECT_SAMPLED, GMC_SELECT_DENSE = 0, 1
STAT_NAMES = ["steps", "pairs", "nnz", "union", "changed", "fallbacks", "nonfinite", "reserved"]
GMC_STAT_COUNT = 8
KERNELS = ["accumulate", "rbgs_step", "sample", "select", "dense_select", "compact",
           "aggregate", "rbgs_pick", "detach", "other"]

_c_p = ctypes.c_void_p
_i64 = ctypes.c_int64
_i32 = ctypes.c_int32
_u64 = ctypes.c_uint64
_f32 = ctypes.c_float
_f64 = ctypes.c_double

# name -> (restype, argtypes)
_SIGNATURES = {
    "gmc_create": (ctypes.c_int, [ctypes.POINTER(_c_p), _i64, _i32, _f32, _f32, _i32, _f64, _i64]),
    "gmc_destroy": (None, [_c_p]),
    "gmc_set_lambda": (ctypes.c_int, [_c_p, _f32]),
    "gmc_set_rbgs_mode": (ctypes.c_int, [_c_p, _i32]),
    "gmc_set_seed": (ctypes.c_int, [_c_p, _u64]),
    "gmc_set_eta": (ctypes.c_int, [_c_p, _f32]),
    "gmc_set_select_mode": (ctypes.c_int, [_c_p, _i32]),
    "gmc_set_variant": (ctypes.c_int, [_c_p, _i32]),
    "gmc_profile_kernels": (ctypes.c_int, [_c_p, ctypes.c_uint32]),
    "gmc_step_bf16": (ctypes.c_int, [_c_p, _c_p, _c_p]),
    "gmc_step_host_bf16": (ctypes.c_int, [_c_p, _c_p, _c_p, _c_p]),
    "gmc_state_bytes": (_i64, [_c_p]),
    "gmc_save_state": (ctypes.c_int, [_c_p, _c_p, _i64]),
    "gmc_load_state": (ctypes.c_int, [_c_p, _c_p, _i64]),
    "gmc_set_detach_output": (ctypes.c_int, [_c_p, _c_p, _i64]),
    "gmc_set_params": (ctypes.c_int, [_c_p, _c_p, _c_p]),
    "gmc_step": (ctypes.c_int, [_c_p, _c_p, _c_p]),
    "gmc_step_host": (ctypes.c_int, [_c_p, _c_p, _c_p, _c_p]),
    "gmc_get_params": (ctypes.c_int, [_c_p, _c_p, _c_p]),
    "gmc_get_residual": (ctypes.c_int, [_c_p, _i32, _c_p, _c_p]),
    "gmc_get_selected": (ctypes.c_int, [_c_p, _i32, _c_p, _c_p, _i64, ctypes.POINTER(_i64), _c_p]),
    "gmc_selected_capacity": (_i64, [_c_p]),
    "gmc_get_worker_params": (ctypes.c_int, [_c_p, _i32, _c_p, _c_p]),
    "gmc_get_stats": (ctypes.c_int, [_c_p, ctypes.POINTER(_u64), _i32, ctypes.POINTER(_f64)]),
    "gmc_check": (ctypes.c_int, [_c_p]),
    "gmc_profile_enable": (ctypes.c_int, [_c_p, _i32]),
    "gmc_profile_read": (ctypes.c_int, [_c_p, _i32, ctypes.POINTER(_f64), ctypes.POINTER(_i64),
                                        ctypes.POINTER(_f64)]),
    "gmc_kernel_name": (ctypes.c_char_p, [_i32]),
    "gmc_strerror": (ctypes.c_char_p, [ctypes.c_int]),
    "gmc_topk_noalloc": (ctypes.c_int, [_c_p, _i64, _i64, _c_p, _c_p, _c_p]),
    "gmc_test_fail_alloc": (_i64, [_i64]),
    "gmc_test_withhold_copy": (ctypes.c_int, [_c_p, _i64, _i32, _u64]),
}

_lib = None


def load() -> ctypes.CDLL:
    """Load libgmc.so (built in-tree); raise ImportError if it is missing."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"{LIB_PATH} is not built; run `python -m paper_1905_12948_gb300.build`")
        lib = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib


def exported_symbols():
    return list(_SIGNATURES)


class GMCError(RuntimeError):
    def __init__(self, status: int, what: str = ""):
        msg = load().gmc_strerror(status).decode()
        super().__init__(f"{what}: {msg} (status {status})" if what else msg)
        self.status = status


def _check(status: int, what: str) -> None:
    if status != GMC_OK:
        raise GMCError(status, what)


def _stream_ptr(stream) -> int:
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream)


def _dev_ptr(t, dtype, name: str) -> int:
    import torch
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype or not t.is_contiguous():
        raise TypeError(f"{name} must be a contiguous {dtype} tensor")
    return t.data_ptr()


class GMC:
    """One GMC / GMC+ handle (Alg. 1 / Alg. 2) for K workers on one GPU."""

    def __init__(self, d: int, K: int, beta: float, eta: float, compressor: str = "topk",
                 ratio: float = 0.01, block: int = 4096, lam: Optional[float] = None,
                 seed: int = 0, per_worker: bool = False, select_mode: str = "sampled",
                 variant: str = "gmc", device=None):
        import torch
        self.torch = torch
        self.lib = load()
        self.d, self.K = int(d), int(K)
        self.compressor = compressor
        self.device = torch.device(device if device is not None else "cuda")
        comp = {"topk": GMC_TOPK, "rbgs": GMC_RBGS, "topk_approx": GMC_TOPK_APPROX}[compressor]
        h = _c_p()
        with torch.cuda.device(self.device):
            _check(self.lib.gmc_create(ctypes.byref(h), self.d, self.K, beta, eta, comp,
                                       float(ratio), int(block)), "gmc_create")
        self.h = h
        if variant != "gmc":
            with torch.cuda.device(self.device):
                _check(self.lib.gmc_set_variant(h, VARIANTS[variant]), "gmc_set_variant")
        if lam is not None:
            _check(self.lib.gmc_set_lambda(h, lam), "gmc_set_lambda")
        _check(self.lib.gmc_set_seed(h, int(seed) & ((1 << 64) - 1)), "gmc_set_seed")
        _check(self.lib.gmc_set_rbgs_mode(h, int(bool(per_worker))), "gmc_set_rbgs_mode")
        mode = {"sampled": GMC_SELECT_SAMPLED, "dense": GMC_SELECT_DENSE}[select_mode]
        _check(self.lib.gmc_set_select_mode(h, mode), "gmc_set_select_mode")
        self._detach = None

    def close(self) -> None:
        if getattr(self, "h", None):
            self.lib.gmc_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- configuration ------------------------------------------------------
    def set_eta(self, eta: float) -> None:
        _check(self.lib.gmc_set_eta(self.h, eta), "gmc_set_eta")

    def set_lambda(self, lam: float) -> None:
        _check(self.lib.gmc_set_lambda(self.h, lam), "gmc_set_lambda")

    def set_detach_output(self, out) -> None:
        """Write w_{t+1,k} into out (K x d float32 CUDA tensor) every step; None disables."""
        if out is None:
            _check(self.lib.gmc_set_detach_output(self.h, None, 0), "gmc_set_detach_output")
        else:
            ptr = _dev_ptr(out, self.torch.float32, "out")
            _check(self.lib.gmc_set_detach_output(self.h, ptr, out.stride(0)), "gmc_set_detach_output")
        self._detach = out

    # -- state and steps ----------------------------------------------------
    def set_params(self, w0, stream=None) -> None:
        _check(self.lib.gmc_set_params(self.h, _dev_ptr(w0, self.torch.float32, "w0"),
                                       _stream_ptr(stream)), "gmc_set_params")

    def step(self, grads, stream=None) -> None:
        """One step from device gradients: a K x d float32 CUDA tensor, or a
        bfloat16 one (gmc_step_bf16: widened exactly, half the bytes)."""
        if tuple(grads.shape) != (self.K, self.d):
            raise ValueError("grads must have shape (K, d)")
        if grads.dtype == self.torch.bfloat16:
            _check(self.lib.gmc_step_bf16(self.h, _dev_ptr(grads, self.torch.bfloat16, "grads"),
                                          _stream_ptr(stream)), "gmc_step_bf16")
            return
        _check(self.lib.gmc_step(self.h, _dev_ptr(grads, self.torch.float32, "grads"),
                                 _stream_ptr(stream)), "gmc_step")

    def step_host(self, grads_host, stats_host=None, stream=None) -> None:
        """One step from host gradients (pinned CPU float32 or bfloat16 tensor
        K x d); the step's counters land in stats_host (pinned CPU int64 tensor of 8)."""
        t = grads_host
        if t.is_cuda or t.dtype not in (self.torch.float32, self.torch.bfloat16) or not t.is_contiguous():
            raise TypeError("grads_host must be a contiguous float32 or bfloat16 CPU tensor")
        if tuple(t.shape) != (self.K, self.d):
            raise ValueError("grads_host must have shape (K, d)")
        sp = stats_host.data_ptr() if stats_host is not None else None
        fn = self.lib.gmc_step_host_bf16 if t.dtype == self.torch.bfloat16 else self.lib.gmc_step_host
        _check(fn(self.h, t.data_ptr(), sp, _stream_ptr(stream)), "gmc_step_host")

    # -- outputs --------------------------------------------------------------
    def params(self, stream=None):
        out = self.torch.empty(self.d, dtype=self.torch.float32, device=self.device)
        _check(self.lib.gmc_get_params(self.h, out.data_ptr(), _stream_ptr(stream)), "gmc_get_params")
        return out

    def residual(self, k: int, stream=None):
        out = self.torch.empty(self.d, dtype=self.torch.float32, device=self.device)
        _check(self.lib.gmc_get_residual(self.h, k, out.data_ptr(), _stream_ptr(stream)),
               "gmc_get_residual")
        return out

    def selected(self, k: int, stream=None) -> Tuple[object, object]:
        """(indices int64, values float32) of worker k's last C(.), ascending index."""
        cap = int(self.lib.gmc_selected_capacity(self.h))
        idx = self.torch.empty(max(cap, 1), dtype=self.torch.int32, device=self.device)
        val = self.torch.empty(max(cap, 1), dtype=self.torch.float32, device=self.device)
        n = _i64()
        _check(self.lib.gmc_get_selected(self.h, k, idx.data_ptr(), val.data_ptr(), cap,
                                         ctypes.byref(n), _stream_ptr(stream)), "gmc_get_selected")
        return idx[: n.value].to(self.torch.int64), val[: n.value]

    def worker_params(self, k: int, stream=None):
        out = self.torch.empty(self.d, dtype=self.torch.float32, device=self.device)
        _check(self.lib.gmc_get_worker_params(self.h, k, out.data_ptr(), _stream_ptr(stream)),
               "gmc_get_worker_params")
        return out

    def stats(self) -> dict:
        arr = (_u64 * GMC_STAT_COUNT)()
        rcc = _f64()
        _check(self.lib.gmc_get_stats(self.h, arr, GMC_STAT_COUNT, ctypes.byref(rcc)), "gmc_get_stats")
        out = {name: int(arr[i]) for i, name in enumerate(STAT_NAMES[:7])}
        out["rcc"] = rcc.value
        return out

    def save_state(self):
        """The handle's state between steps (gmc_save_state) as a numpy uint8 array."""
        import numpy as np
        n = int(self.lib.gmc_state_bytes(self.h))
        buf = np.empty(n, np.uint8)
        _check(self.lib.gmc_save_state(self.h, buf.ctypes.data, n), "gmc_save_state")
        return buf

    def load_state(self, buf) -> None:
        """Continue from a state saved by save_state (gmc_load_state)."""
        import numpy as np
        buf = np.ascontiguousarray(buf, np.uint8)
        _check(self.lib.gmc_load_state(self.h, buf.ctypes.data, buf.size), "gmc_load_state")

    def check(self) -> int:
        return int(self.lib.gmc_check(self.h))

    # -- profiling ----------------------------------------------------------
    def profile(self, on: bool = True, kernels=None) -> None:
        """Bracket the step's launches with events (all kernels, or the named ones)."""
        mask = 0xFFFFFFFF if kernels is None else sum(1 << KERNELS.index(k) for k in kernels)
        _check(self.lib.gmc_profile_kernels(self.h, mask), "gmc_profile_kernels")
        _check(self.lib.gmc_profile_enable(self.h, int(on)), "gmc_profile_enable")

    def profile_mask(self, kernels=None) -> None:
        """Choose the launches bracketed while profiling is on (all, or the named ones)."""
        mask = 0xFFFFFFFF if kernels is None else sum(1 << KERNELS.index(k) for k in kernels)
        _check(self.lib.gmc_profile_kernels(self.h, mask), "gmc_profile_kernels")

    def profile_read(self) -> dict:
        out = {}
        for i, name in enumerate(KERNELS):
            ms, n, b = _f64(), _i64(), _f64()
            _check(self.lib.gmc_profile_read(self.h, i, ctypes.byref(ms), ctypes.byref(n),
                                             ctypes.byref(b)), "gmc_profile_read")
            if n.value:
                out[name] = {"ms": ms.value, "launches": n.value, "bytes": b.value}
        return out


# C-ABI names, re-exported for callers that prefer the flat interface.
def __getattr__(name):
    if name.startswith("gmc_") and name in _SIGNATURES:
        return getattr(load(), name)
    raise AttributeError(name)
