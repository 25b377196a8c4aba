"""Helpers for the GPU-vs-oracle parity tests: run both on the same seeded
inputs and compare every step -- selected indices bit-exact, values, w and e
bitwise and within the stated fp32 bar (1e-6 relative, 1e-7 absolute)."""
import numpy as np

import oracle
from oracle import cref

RTOL, ATOL = 1e-6, 1e-7


def bits(a):
    return np.ascontiguousarray(a, np.float32).view(np.uint32)


def assert_fp32_state(got, want, what):
    got = np.asarray(got, np.float32)
    want = np.asarray(want, np.float32)
    np.testing.assert_allclose(got, want, rtol=RTOL, atol=ATOL, err_msg=what)
    diff = np.flatnonzero(bits(got) != bits(want))
    assert diff.size == 0, f"{what}: {diff.size} values differ bitwise, first at {diff[:5]}"


class Pair:
    """A CUDA handle and an oracle instance fed identical inputs."""

    def __init__(self, d, K, beta, eta, compressor="topk", ratio=0.01, block=4096, lam=None,
                 seed=0, per_worker=False, select_mode="sampled", w0=None, device="cuda",
                 variant="gmc", ref="numpy"):
        import torch
        from paper_1905_12948_gb300 import GMC
        self.torch = torch
        self.d, self.K = d, K
        self.dev = torch.device(device)
        lam_or = (0.5 if compressor == "rbgs" else 0.0) if lam is None else lam
        self.gpu = GMC(d, K, beta, eta, compressor=compressor, ratio=ratio, block=block, lam=lam,
                       seed=seed, per_worker=per_worker, select_mode=select_mode, device=self.dev,
                       variant=variant)
        # the numpy oracle, or the C++ one (Alg. 1 / Alg. 2 with top-s or RBGS;
        # fast enough for whole trajectories at full size)
        make = oracle.GMC if ref == "numpy" else cref.CGMC
        self.ref = make(d, K, beta, eta, compressor=compressor, ratio=ratio, block=block,
                        lam=lam_or, seed=seed, per_worker=per_worker, variant=variant)
        if w0 is None:
            w0 = (np.random.default_rng(seed + 17).standard_normal(d) * 0.01).astype(np.float32)
        self.gpu.set_params(torch.from_numpy(w0).to(self.dev))
        self.ref.set_params(w0)

    def step(self, g, grads_dev=None):
        if grads_dev is None:
            grads_dev = self.torch.from_numpy(np.ascontiguousarray(g)).to(self.dev)
        self.gpu.step(grads_dev)
        return self.ref.step(g)

    def compare(self, r, residuals=True, workers=None, state=True):
        """Selections of step r; then, if `state`, w and the residuals (reading
        them applies an aggregation the library may have left pending)."""
        ks = range(self.K) if workers is None else workers
        for k in ks:
            idx, val = self.gpu.selected(k)
            idx = idx.cpu().numpy()
            assert np.array_equal(idx, r.supports[k]), (
                f"worker {k}: selected indices differ "
                f"({np.setdiff1d(idx, r.supports[k])[:5]} vs {np.setdiff1d(r.supports[k], idx)[:5]})")
            assert np.array_equal(bits(val.cpu().numpy()), bits(r.values[k])), f"worker {k}: values"
        if not state:
            return
        assert_fp32_state(self.gpu.params().cpu().numpy(), self.ref.w, "w")
        if residuals:
            for k in ks:
                assert_fp32_state(self.gpu.residual(k).cpu().numpy(), self.ref.e[k], f"e[{k}]")

    def compare_stats(self):
        s = self.gpu.stats()
        tot = self.ref.totals
        for key in ("steps", "pairs", "nnz", "union", "changed"):
            assert s[key] == tot[key], (key, s[key], tot[key])
        assert abs(s["rcc"] - self.ref.rcc()) <= 1e-12 * max(1.0, self.ref.rcc())
        return s
