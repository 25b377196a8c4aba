"""ctypes wrapper of the C++ oracle (``gmc_ref.cpp``): Algorithm 1 / 2 with the
top-s and RBGS compressors, written out with dense arrays, one worker per
thread.

TEST INFRASTRUCTURE, like the numpy oracle next to it: only the tests,
``__graft_entry__.smoke()`` and the CPU baseline / reference arm of
``bench.py`` may import this module. It shares no code with the CUDA path.

The C++ oracle states the same rules and readings as ``gmc_oracle.GMC`` (see
that module's header) for the method's own step -- GMC and GMC+, exact top-s
and RBGS -- in a second, independent implementation that is fast enough to
follow the full-size workloads over whole trajectories. The pins of
``tests/test_oracle_pins.py`` run on both.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "gmc_ref.cpp")
LIB = os.path.join(HERE, "libgmcref.so")
# IEEE fp32 arithmetic as written: no FMA contraction, no fast-math
CXXFLAGS = ["-O2", "-std=c++17", "-fPIC", "-shared", "-pthread", "-ffp-contract=off", "-fno-fast-math"]

_lib = None


def build(force: bool = False) -> str:
    """Compile libgmcref.so next to its source when missing or older than it."""
    if force or not os.path.exists(LIB) or os.path.getmtime(LIB) < os.path.getmtime(SRC):
        tmp = LIB + f".{os.getpid()}.tmp"
        subprocess.run(["g++", *CXXFLAGS, "-o", tmp, SRC], check=True)
        os.replace(tmp, LIB)
    return LIB


def load() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(LIB)
        vp, i64, i32, u64, f32, f64 = (ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32,
                                       ctypes.c_uint64, ctypes.c_float, ctypes.c_double)
        sig = {
            "gmcref_create": (vp, [i64, i32, f32, f32, i32, f64, i64, f32, u64, i32, i32]),
            "gmcref_destroy": (None, [vp]),
            "gmcref_threads": (i32, [vp]),
            "gmcref_set_params": (ctypes.c_int, [vp, vp]),
            "gmcref_set_eta": (ctypes.c_int, [vp, f32]),
            "gmcref_step": (ctypes.c_int, [vp, vp]),
            "gmcref_support_size": (i64, [vp, i32]),
            "gmcref_support": (ctypes.c_int, [vp, i32, vp, vp]),
            "gmcref_w": (vp, [vp]),
            "gmcref_e": (vp, [vp]),
            "gmcref_worker_params": (ctypes.c_int, [vp, i32, vp]),
            "gmcref_totals": (ctypes.c_int, [vp, vp]),
            "gmcref_top_s": (ctypes.c_int, [vp, i64, i64, vp]),
            "gmcref_rbgs_blocks": (ctypes.c_int, [u64, i64, u64, i64, i64, vp]),
            "gmcref_splitmix64_next": (u64, [ctypes.POINTER(u64)]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(lib, name)
            fn.restype, fn.argtypes = res, args
        _lib = lib
    return _lib


def top_s_support(x: np.ndarray, s: int) -> np.ndarray:
    """Top-s support of one vector (ascending), from the C++ oracle."""
    x = np.ascontiguousarray(x, np.float32)
    if not 1 <= s <= x.size:
        raise ValueError("s must be in [1, d]")
    out = np.empty(s, np.int64)
    assert load().gmcref_top_s(x.ctypes.data, x.size, s, out.ctypes.data) == 0
    return out


def rbgs_blocks(seed: int, t: int, stream: int, nb: int, m: int) -> np.ndarray:
    """The m blocks of step t's stream (0: shared, k + 1: worker k), ascending."""
    out = np.empty(m, np.int64)
    assert load().gmcref_rbgs_blocks(seed, t, stream, nb, m, out.ctypes.data) == 0
    return out


def splitmix64_sequence(seed: int, n: int):
    st = ctypes.c_uint64(seed & ((1 << 64) - 1))
    return [int(load().gmcref_splitmix64_next(ctypes.byref(st))) for _ in range(n)]


class StepResult:
    """The selections of one step: supports (ascending int64) and values per
    worker; with `keep_half`, also e_{t+1/2,k} (the residual after the step
    with the sent values put back)."""

    def __init__(self, supports, values, e_half=None):
        self.supports = supports
        self.values = values
        self.e_half = e_half


class CGMC:
    """Algorithm 1 (GMC) / Algorithm 2 (GMC+) for K workers: the C++ oracle,
    with the interface of ``gmc_oracle.GMC`` for the top-s and RBGS steps."""

    def __init__(self, d: int, K: int, beta: float, eta: float, compressor: str = "topk",
                 ratio: float = 0.01, block: int = 4096, lam: float = 0.0, seed: int = 0,
                 per_worker: bool = False, variant: str = "gmc", threads: int = 0,
                 keep_half: bool = False):
        if variant != "gmc" or compressor not in ("topk", "rbgs"):
            raise ValueError("the C++ oracle states Alg. 1 / Alg. 2 with top-s or RBGS only")
        self.lib = load()
        self.d, self.K = int(d), int(K)
        self.compressor = compressor
        self.keep_half = keep_half
        # the fp32 constants, as the oracle forms them (for rounding budgets in tests)
        self.beta, self.lam = np.float32(beta), np.float32(lam)
        self.eta = np.float32(eta)
        self.c = np.float32(self.beta / self.eta)
        self.h = self.lib.gmcref_create(self.d, self.K, beta, eta, 0 if compressor == "topk" else 1,
                                        float(ratio), int(block), float(lam),
                                        int(seed) & ((1 << 64) - 1), int(bool(per_worker)), int(threads))
        if not self.h:
            raise ValueError("invalid oracle arguments")
        self.threads = int(self.lib.gmcref_threads(self.h))

    def __del__(self):
        h, self.h = getattr(self, "h", None), None
        if h:
            self.lib.gmcref_destroy(h)

    def set_params(self, w0: np.ndarray) -> None:
        w0 = np.ascontiguousarray(w0, np.float32)
        if w0.shape != (self.d,):
            raise ValueError("w0 must have shape (d,)")
        assert self.lib.gmcref_set_params(self.h, w0.ctypes.data) == 0

    def set_eta(self, eta: float) -> None:
        assert self.lib.gmcref_set_eta(self.h, eta) == 0
        self.eta = np.float32(eta)
        self.c = np.float32(self.beta / self.eta)

    def step(self, grads: np.ndarray) -> StepResult:
        g = np.ascontiguousarray(grads, np.float32)
        if g.shape != (self.K, self.d):
            raise ValueError("grads must have shape (K, d)")
        assert self.lib.gmcref_step(self.h, g.ctypes.data) == 0, "set_params first"
        sup, val = [], []
        for k in range(self.K):
            n = int(self.lib.gmcref_support_size(self.h, k))
            idx = np.empty(n, np.int64)
            v = np.empty(n, np.float32)
            assert self.lib.gmcref_support(self.h, k, idx.ctypes.data, v.ctypes.data) == 0
            sup.append(idx)
            val.append(v)
        half = None
        if self.keep_half:
            half = self.e.copy()
            for k in range(self.K):
                half[k, sup[k]] = val[k]
        return StepResult(sup, val, half)

    @property
    def w(self) -> np.ndarray:
        """w_t, a view of the oracle's array (valid until set_params)."""
        p = self.lib.gmcref_w(self.h)
        return np.ctypeslib.as_array(ctypes.cast(p, ctypes.POINTER(ctypes.c_float)), (self.d,))

    @property
    def e(self) -> np.ndarray:
        """e_{t,k} for every k (K x d), a view of the oracle's array."""
        p = self.lib.gmcref_e(self.h)
        return np.ctypeslib.as_array(ctypes.cast(p, ctypes.POINTER(ctypes.c_float)), (self.K, self.d))

    def worker_params(self, k: int) -> np.ndarray:
        out = np.empty(self.d, np.float32)
        assert self.lib.gmcref_worker_params(self.h, k, out.ctypes.data) == 0
        return out

    @property
    def totals(self) -> dict:
        arr = np.zeros(5, np.uint64)
        assert self.lib.gmcref_totals(self.h, arr.ctypes.data) == 0
        return dict(zip(("steps", "pairs", "nnz", "union", "changed"), (int(x) for x in arr)))

    def rcc(self) -> float:
        """Relative communication cost (Sec. 5), halved for RBGS (Sec. 5.2)."""
        tot = self.totals
        if tot["steps"] == 0:
            return 0.0
        r = (self.K * tot["changed"] + tot["nnz"]) / (self.d * self.K * tot["steps"])
        return r / 2 if self.compressor == "rbgs" else r
