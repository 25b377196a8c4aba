"""GPU-vs-oracle parity of the approximate top-s compressor (Sec. 5.1): the
shared stratified sample, the exact sampled threshold, every component at or
above it sent (the count varies by worker and step), the limit beyond which
the exact top is sent, on both dense passes, with deferred and eager
aggregation."""
import numpy as np
import pytest

import oracle
from parity_util import Pair

pytestmark = pytest.mark.gpu


def _grads(rng, K, d):
    return (rng.standard_normal((K, d)) * np.exp(rng.uniform(-3, 0, size=d))).astype(np.float32)


def _check_counts(p, r):
    for k in range(p.K):
        idx, _ = p.gpu.selected(k)
        assert idx.numel() == r.supports[k].size


@pytest.mark.parametrize("d,K,ratio", [(50_000, 4, 0.01), (100, 2, 0.5), (99, 3, 0.01),
                                       (333_337, 5, 1 / 1024)])
def test_approx_load_store_pass(d, K, ratio):
    """Below the bulk pass's size: the load/store pass, aggregate each step."""
    rng = np.random.default_rng(d + K)
    p = Pair(d, K, 0.9, 0.1, compressor="topk_approx", ratio=ratio, seed=7)
    for t in range(5):
        r = p.step(_grads(rng, K, d))
        p.compare(r)
        _check_counts(p, r)
    p.compare_stats()
    assert p.gpu.check() == 0


@pytest.mark.parametrize("d,K", [(1_300_001, 8), (4096 * 200, 3), (1_250_003, 1)])
def test_approx_bulk_pass_deferred(d, K):
    """The bulk pass with the aggregation deferred into the next step; the
    selections are compared every step, the state at the end."""
    rng = np.random.default_rng(3 + K)
    p = Pair(d, K, 0.9, 0.05, compressor="topk_approx", ratio=1 / 1024, seed=11)
    for t in range(4):
        r = p.step(_grads(rng, K, d))
        p.compare(r, state=(t == 3))
    s = p.compare_stats()
    assert s["fallbacks"] == 0
    assert p.gpu.check() == 0


def test_approx_many_workers_and_eta_schedule():
    """More workers than the bulk pass takes, and eta changed between steps."""
    d, K = 1_300_001, 20
    rng = np.random.default_rng(21)
    p = Pair(d, K, 0.9, 0.1, compressor="topk_approx", ratio=0.002, seed=2)
    for t in range(3):
        eta = 0.1 * 0.5 * (1 + np.cos(np.pi * t / 6))
        p.gpu.set_eta(eta)
        p.ref.set_eta(eta)
        r = p.step(_grads(rng, K, d))
        p.compare(r, residuals=(t == 2))
    p.compare_stats()
    assert p.gpu.check() == 0


@pytest.mark.parametrize("d", [20_000, 1_300_001])
def test_approx_limit_takes_exact_top(d):
    """All-zero accumulators: theta is the zero key and every component
    reaches it, so the limit applies and the exact top (the lowest indices)
    is sent, through the dense path, on both passes."""
    import torch
    K = 2
    p = Pair(d, K, 0.9, 0.1, compressor="topk_approx", ratio=0.001, seed=1,
             w0=np.zeros(d, np.float32))
    zeros = np.zeros((K, d), np.float32)
    r = p.step(zeros)
    p.compare(r)
    for k in range(K):
        np.testing.assert_array_equal(r.supports[k], np.arange(p.ref.limit))
    # then ordinary data: the next selections are threshold sets again
    rng = np.random.default_rng(4)
    for t in range(2):
        r = p.step(_grads(rng, K, d))
        p.compare(r)
    s = p.compare_stats()
    assert s["fallbacks"] >= K
    assert p.gpu.check() == 0
    del torch


def test_approx_ties_all_sent():
    """Values from a small set: many components equal theta; all are sent."""
    d, K = 1_300_001, 3
    rng = np.random.default_rng(8)
    p = Pair(d, K, 0.0, 0.1, compressor="topk_approx", ratio=0.001, seed=5,
             w0=np.zeros(d, np.float32))
    vals = np.array([-4.0, -3.0, -0.5, -0.25, 0.0, 0.25, 0.5, 3.0, 4.0], np.float32)
    prob = [0.001, 0.0015, 0.2, 0.2, 0.195, 0.2, 0.2, 0.0015, 0.001]
    for t in range(3):
        g = rng.choice(vals, size=(K, d), p=prob)
        r = p.step(g.astype(np.float32))
        p.compare(r, state=(t == 2))
    p.compare_stats()
    assert p.gpu.check() == 0


def test_approx_host_steps_and_gmcplus_detach():
    """Host gradients (in place when page-locked) and the GMC+ detach output."""
    import torch
    d, K = 1_300_001, 4
    rng = np.random.default_rng(9)
    p = Pair(d, K, 0.9, 0.05, compressor="topk_approx", ratio=1 / 1024, seed=3, lam=0.5)
    out = torch.empty((K, d), dtype=torch.float32, device=p.dev)
    p.gpu.set_detach_output(out)
    for t in range(3):
        g = _grads(rng, K, d)
        host = torch.from_numpy(g).pin_memory() if t != 1 else torch.from_numpy(g)
        p.gpu.step_host(host)
        r = p.ref.step(g)
        p.compare(r)
        torch.cuda.synchronize()
        for k in range(K):
            np.testing.assert_array_equal(out[k].cpu().numpy().view(np.uint32),
                                          p.ref.worker_params(k).view(np.uint32))
    p.compare_stats()
    assert p.gpu.check() == 0


def test_approx_count_tracks_ratio_at_vgg_like_scale():
    """Count of one worker's selection near ratio*d (Sec. 5.1's 'approximately
    d/1024') on heavy-tailed synthetic data, and equal to the oracle's."""
    d, K = 4_000_037, 2
    rng = np.random.default_rng(10)
    p = Pair(d, K, 0.9, 0.05, compressor="topk_approx", ratio=1 / 1024, seed=4)
    r = p.step(_grads(rng, K, d))
    p.compare(r)
    for k in range(K):
        assert 0.5 < r.supports[k].size / (d / 1024) < 1.5
    assert r.sample.size == oracle.approx_sample_size(d)


def test_approx_rejects_dense_engine():
    from paper_1905_12948_gb300 import GMC
    from paper_1905_12948_gb300.gmc import GMCError
    with pytest.raises(GMCError):
        GMC(1000, 2, 0.9, 0.1, compressor="topk_approx", ratio=0.01, select_mode="dense")
