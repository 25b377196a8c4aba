"""Checkpoint / resume through the C ABI: a trajectory saved mid-run (with an
aggregation still pending, for the deferred top-k path) and loaded into a new
handle continues exactly as the oracle's uninterrupted run, for every
compressor, both dense passes and every variant of the step (with their extra
state: Alg. 3's server momentum, the workers' local momentum); malformed or
mismatched states are refused."""
import numpy as np
import pytest

from parity_util import Pair

pytestmark = pytest.mark.gpu


def _grads(rng, K, d):
    return (rng.standard_normal((K, d)) * np.exp(rng.uniform(-3, 0, size=d))).astype(np.float32)


def _fresh(p, **kw):
    from paper_1905_12948_gb300 import GMC
    return GMC(p.d, p.K, float(p.ref.beta), float(p.ref.eta), device=p.dev, **kw)


CASES = [
    dict(compressor="topk", d=1_300_001, K=4, ratio=0.002),               # bulk pass, deferred
    dict(compressor="topk", d=1_300_001, K=6, ratio=0.002),               # and its one-tile pipeline
    dict(compressor="topk", d=50_003, K=3, ratio=0.01),                   # load/store pass
    dict(compressor="topk_approx", d=1_300_001, K=3, ratio=1 / 1024),
    dict(compressor="rbgs", d=4096 * 160 + 3, K=5, ratio=0.05, block=4096, lam=0.5),
    dict(compressor="rbgs", d=70_001, K=3, ratio=0.1, block=1000, lam=0.5, per_worker=True),
    dict(compressor="topk", d=1_300_001, K=3, ratio=0.002, variant="server_momentum"),
    dict(compressor="topk", d=1_300_001, K=3, ratio=0.002, variant="lr_in_residual"),
    dict(compressor="topk", d=1_300_001, K=3, ratio=0.002, variant="local_momentum"),
    dict(compressor="topk", d=1_300_001, K=7, ratio=0.002, variant="local_momentum"),
    dict(compressor="topk_approx", d=50_003, K=2, ratio=0.01, variant="local_momentum_mfm"),
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: "-".join(str(v) for v in c.values()))
def test_resume_continues_the_trajectory(case):
    case = dict(case)
    d, K = case.pop("d"), case.pop("K")
    rng = np.random.default_rng(d + K)
    p = Pair(d, K, 0.9, 0.1, seed=13, **case)
    for t in range(3):
        p.compare(p.step(_grads(rng, K, d)), state=(t == 2 and case["compressor"] != "topk"))
    state = p.gpu.save_state()
    assert state.size == p.gpu.lib.gmc_state_bytes(p.gpu.h)
    old = p.gpu
    p.gpu = _fresh(p, compressor=case["compressor"], ratio=case["ratio"],
                   block=case.get("block", 4096), variant=case.get("variant", "gmc"))
    p.gpu.load_state(state)
    with pytest.raises(Exception):
        p.gpu.selected(0)  # no selection since the restore
    # the saved handle itself continues too, in step with the restored one
    for t in range(3):
        g = _grads(rng, K, d)
        old.step(__import__("torch").from_numpy(g).to(p.dev))
        r = p.step(g)
        p.compare(r, state=(t == 2))
        for k in range(K):
            a, b = old.selected(k), p.gpu.selected(k)
            assert np.array_equal(a[0].cpu().numpy(), b[0].cpu().numpy())
    p.compare_stats()
    assert p.gpu.check() == 0 and old.check() == 0
    np.testing.assert_array_equal(old.params().cpu().numpy().view(np.uint32),
                                  p.gpu.params().cpu().numpy().view(np.uint32))


def test_resume_at_step_zero_and_settings_restored():
    """A state saved before the first step; eta, seed and the step count come
    back with it (they drive the schedule and the random choices)."""
    d, K = 70_001, 3
    rng = np.random.default_rng(2)
    p = Pair(d, K, 0.9, 0.1, compressor="rbgs", ratio=0.1, block=1000, seed=99, lam=0.5)
    p.gpu.set_eta(0.05)
    p.ref.set_eta(0.05)
    state = p.gpu.save_state()
    p.gpu = _fresh(p, compressor="rbgs", ratio=0.1, block=1000, seed=0)  # seed, eta differ
    p.gpu.load_state(state)
    for t in range(2):
        p.compare(p.step(_grads(rng, K, d)))
    p.compare_stats()


def test_load_refuses_mismatched_or_malformed_states():
    from paper_1905_12948_gb300 import GMC
    from paper_1905_12948_gb300.gmc import GMCError
    import torch
    a = GMC(10_000, 2, 0.9, 0.1, ratio=0.01)
    a.set_params(torch.zeros(10_000, device="cuda"))
    a.step(torch.ones((2, 10_000), device="cuda"))
    s = a.save_state()
    for other in (GMC(10_001, 2, 0.9, 0.1, ratio=0.01), GMC(10_000, 3, 0.9, 0.1, ratio=0.01),
                  GMC(10_000, 2, 0.9, 0.1, ratio=0.02), GMC(10_000, 2, 0.9, 0.1, ratio=0.01,
                                                            compressor="topk_approx"),
                  GMC(10_000, 2, 0.9, 0.1, ratio=0.01, variant="lr_in_residual")):
        with pytest.raises(GMCError):
            other.load_state(s)
    b = GMC(10_000, 2, 0.9, 0.1, ratio=0.01)
    with pytest.raises(GMCError):
        b.load_state(s[:-1])
    bad = s.copy()
    bad[0] ^= 1
    with pytest.raises(GMCError):
        b.load_state(bad)
    b.load_state(s)
    assert np.array_equal(b.params().cpu().numpy(), a.params().cpu().numpy())
