"""GPU-vs-oracle parity through the C ABI on seeded synthetic inputs, at sizes
the oracle runs in seconds: ragged tails, misaligned gradient rows, forced
ties, both selection engines, RBGS in both modes with GMC+, and edge cases."""
import numpy as np
import pytest

import workloads
from parity_util import Pair, assert_fp32_state, bits

pytestmark = pytest.mark.gpu


def _tie_grads(rng, K, d, scale=1.0):
    return (rng.choice([-2.0, -1.0, -0.0, 0.0, 1.0, 2.0], size=(K, d)) * scale).astype(np.float32)


@pytest.mark.parametrize("select_mode", ["sampled", "dense"])
@pytest.mark.parametrize("d,K,ratio", [(1000, 3, 0.05), (4099, 2, 0.01), (1, 1, 0.5), (7, 2, 1.0)])
def test_topk_forced_ties(select_mode, d, K, ratio):
    rng = np.random.default_rng(d + K)
    p = Pair(d, K, 0.9, 0.1, ratio=ratio, select_mode=select_mode, seed=3)
    for t in range(6):
        r = p.step(_tie_grads(rng, K, d, scale=0.5 ** t))
        p.compare(r)
    p.compare_stats()
    assert p.gpu.check() == 0


@pytest.mark.parametrize("wl_name", ["mlp65k", "resnet20"])
def test_topk_workload_trajectory(wl_name):
    """Whole configured trajectories of the two small workloads."""
    wl = workloads.workload(wl_name)
    gen = workloads.NumpyGradients(wl, seed=0)
    p = Pair(wl.d, wl.K, wl.beta, wl.eta, ratio=wl.ratio, w0=workloads.init_params(wl.d))
    for t in range(wl.steps):
        r = p.step(gen(t))
        p.compare(r, residuals=(t % 10 == 9 or t == wl.steps - 1))
    s = p.compare_stats()
    assert s["fallbacks"] == 0
    assert p.gpu.check() == 0


def test_topk_sampled_and_dense_agree_ragged_large():
    """d above the full-sample size, odd, with misaligned rows: both engines
    give the oracle's result."""
    d, K = 100_003, 5
    rng = np.random.default_rng(5)
    pairs = [Pair(d, K, 0.9, 0.05, ratio=0.003, select_mode=m, seed=1) for m in ("sampled", "dense")]
    for t in range(4):
        g = (rng.standard_normal((K, d)) * np.exp(rng.uniform(-3, 0, size=d))).astype(np.float32)
        for p in pairs:
            p.compare(p.step(g))
    assert pairs[0].gpu.stats()["fallbacks"] == 0
    assert pairs[1].gpu.stats()["fallbacks"] == 4 * K


@pytest.mark.parametrize("offset", [0, 1])
def test_topk_bulk_copy_path(offset):
    """d large enough for the bulk-copy dense pass (tiles of 4096); odd d gives
    rows at every alignment, and offset 1 makes the first row start 4 bytes
    past an aligned address so its bulk copy would begin before the buffer
    (that row is then loaded directly)."""
    import torch
    d, K = 1_300_001, 3
    rng = np.random.default_rng(15 + offset)
    p = Pair(d, K, 0.9, 0.05, ratio=0.002, seed=2)
    for t in range(3):
        g = (rng.standard_normal((K, d)) * np.exp(rng.uniform(-3, 0, size=d))).astype(np.float32)
        buf = torch.empty(K * d + offset, dtype=torch.float32, device=p.dev)
        view = buf[offset:].view(K, d)
        view.copy_(torch.from_numpy(g))
        p.compare(p.step(g, grads_dev=view), residuals=(t == 2))
    assert p.gpu.stats()["fallbacks"] == 0
    assert p.gpu.check() == 0


def test_topk_many_workers_take_load_store_pass():
    """More workers than the bulk pass takes (17..32): the load/store pass at
    a size that would otherwise be bulk, with the aggregate applied each step."""
    d, K = 1_300_001, 20
    rng = np.random.default_rng(17)
    p = Pair(d, K, 0.9, 0.05, ratio=0.001, seed=7)
    for t in range(2):
        g = (rng.standard_normal((K, d)) * np.exp(rng.uniform(-3, 0, size=d))).astype(np.float32)
        p.compare(p.step(g), residuals=(t == 1))
    p.compare_stats()
    assert p.gpu.check() == 0


def test_topk_dense_tiles_unstaged_aggregate():
    """Every coordinate sent by 5 workers: more entries per tile than the
    aggregate stages in shared memory."""
    d, K = 3000, 5
    rng = np.random.default_rng(16)
    p = Pair(d, K, 0.9, 0.1, ratio=1.0)
    for t in range(3):
        p.compare(p.step(rng.standard_normal((K, d)).astype(np.float32)))
    p.compare_stats()


def test_topk_all_zero_gradients_fall_back():
    """Every magnitude ties: the selection is the k lowest indices; above the
    full-sample size the candidate filter overflows and the dense path runs."""
    d, K = 40_000, 2
    p = Pair(d, K, 0.9, 0.1, ratio=0.01, w0=np.zeros(d, np.float32))
    for _ in range(2):
        r = p.step(np.zeros((K, d), np.float32))
        p.compare(r)
        np.testing.assert_array_equal(r.supports[0], np.arange(p.ref.s))
    assert p.gpu.stats()["fallbacks"] == 2 * K


def test_misaligned_gradient_pointer():
    """Gradient rows starting at any 4-byte offset."""
    import torch
    d, K = 3001, 3
    rng = np.random.default_rng(7)
    p = Pair(d, K, 0.9, 0.1, ratio=0.02)
    for t in range(3):
        g = rng.standard_normal((K, d)).astype(np.float32)
        buf = torch.empty(K * d + 1, dtype=torch.float32, device=p.dev)
        view = buf[1:].view(K, d)
        view.copy_(torch.from_numpy(g))
        p.compare(p.step(g, grads_dev=view))


def test_eta_schedule_between_steps():
    """The cosine learning-rate schedule of Sec. 5.1 applied between steps."""
    import math
    d, K = 20_000, 4
    rng = np.random.default_rng(8)
    p = Pair(d, K, 0.9, 0.1, ratio=0.01)
    for t in range(5):
        eta = 0.1 * 0.5 * (1 + math.cos(t * math.pi / 5))
        eta = max(eta, 1e-3)
        p.gpu.set_eta(eta)
        p.ref.set_eta(eta)
        p.compare(p.step(rng.standard_normal((K, d)).astype(np.float32)))


def test_step_host_matches_step():
    import torch
    d, K = 12_345, 3
    rng = np.random.default_rng(9)
    p = Pair(d, K, 0.9, 0.1, ratio=0.01)
    stats = torch.zeros(8, dtype=torch.int64).pin_memory()
    for t in range(3):
        g = rng.standard_normal((K, d)).astype(np.float32)
        p.gpu.step_host(torch.from_numpy(g).pin_memory(), stats)
        r = p.ref.step(g)
        torch.cuda.synchronize()
        p.compare(r)
        assert int(stats[1]) == r.stats["pairs"] and int(stats[3]) == r.stats["union"]
        assert int(stats[4]) == r.stats["changed"] and int(stats[0]) == 1


@pytest.mark.parametrize("per_worker", [False, True])
@pytest.mark.parametrize("d,B,ratio", [(10_000, 64, 0.05), (5_003, 100, 0.1), (4096 * 3 + 5, 4096, 0.5),
                                        # enough tiles for the bulk-copy kernel: odd d (rows at
                                        # every alignment), blocks that straddle tiles, and B = tile
                                        (700_001, 1000, 0.02), (4096 * 160 + 3, 4096, 0.05),
                                        # about five tiles per CTA: the later ones claimed
                                        (4096 * 152 * 5 + 77, 4096, 0.02)])
def test_rbgs_gmcplus(per_worker, d, B, ratio):
    import torch
    K = 4
    rng = np.random.default_rng(d + B)
    p = Pair(d, K, 0.9, 0.1, compressor="rbgs", ratio=ratio, block=B, lam=0.5, seed=11,
             per_worker=per_worker)
    out = torch.zeros((K, d), dtype=torch.float32, device=p.dev)
    p.gpu.set_detach_output(out)
    for t in range(5):
        r = p.step(rng.standard_normal((K, d)).astype(np.float32))
        p.compare(r)
        host = out.cpu().numpy()
        for k in range(K):
            assert_fp32_state(host[k], p.ref.worker_params(k), f"w_(t,{k})")
            assert_fp32_state(p.gpu.worker_params(k).cpu().numpy(), p.ref.worker_params(k), "detach")
    p.compare_stats()


def test_topk_gmcplus_detach():
    d, K = 5000, 3
    rng = np.random.default_rng(12)
    p = Pair(d, K, 0.9, 0.1, ratio=0.02, lam=0.3)
    for t in range(3):
        p.compare(p.step(rng.standard_normal((K, d)).astype(np.float32)))
        for k in range(K):
            assert_fp32_state(p.gpu.worker_params(k).cpu().numpy(), p.ref.worker_params(k), "detach")


def test_nonfinite_reported():
    d, K = 2000, 2
    p = Pair(d, K, 0.9, 0.1, ratio=0.01)
    g = np.ones((K, d), np.float32)
    g[1, 77] = np.nan
    g[0, 5] = np.inf
    p.gpu.step(p.torch.from_numpy(g).to(p.dev))
    assert p.gpu.check() == 4  # GMC_ENONFINITE
    assert p.gpu.stats()["nonfinite"] == 2


def test_errors_on_bad_calls():
    import torch
    from paper_1905_12948_gb300 import GMC, GMCError
    h = GMC(100, 2, 0.9, 0.1)
    with pytest.raises(GMCError):  # before set_params
        h.step(torch.zeros((2, 100), device="cuda"))
    with pytest.raises(ValueError):
        h.step(torch.zeros((3, 100), device="cuda"))
    with pytest.raises(GMCError):
        GMC(0, 2, 0.9, 0.1)
    with pytest.raises(GMCError):
        h.set_lambda(2.0)
