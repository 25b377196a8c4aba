"""GPU-vs-oracle parity of the variants of the step: the appendix's Alg. 3
(momentum on the server, a dense update of w every step) and Alg. 4
(learning rate inside the residual), and the local-momentum baseline of
Sec. 2.3 with error feedback (DGC without / with momentum factor masking),
with both top-k compressors, on the load/store and bulk passes, with the
learning-rate schedule between steps and host steps."""
import numpy as np
import pytest

from parity_util import Pair

pytestmark = pytest.mark.gpu

VARIANTS = ["server_momentum", "lr_in_residual", "local_momentum", "local_momentum_mfm"]
EAGER = ("server_momentum", "local_momentum_mfm")  # these aggregate every step at once


def _grads(rng, K, d):
    return (rng.standard_normal((K, d)) * np.exp(rng.uniform(-3, 0, size=d))).astype(np.float32)


@pytest.mark.parametrize("variant", VARIANTS)
@pytest.mark.parametrize("compressor", ["topk", "topk_approx"])
@pytest.mark.parametrize("d,K", [(50_003, 4), (1_300_001, 3)])
def test_variant_parity(variant, compressor, d, K):
    rng = np.random.default_rng(d + K + len(variant))
    p = Pair(d, K, 0.9, 0.1, compressor=compressor, ratio=0.002, seed=6, variant=variant)
    for t in range(4):
        r = p.step(_grads(rng, K, d))
        # the others defer their aggregation on the bulk pass: read the state at the end
        p.compare(r, state=(variant in EAGER or d < 1_000_000 or t == 3))
    s = p.compare_stats()
    assert s["fallbacks"] == 0
    assert p.gpu.check() == 0


@pytest.mark.parametrize("variant", VARIANTS)
def test_variant_eta_schedule_and_host_steps(variant):
    """The cosine schedule of Sec. 5.1 between steps (Alg. 4 scales each
    step's gradient by that step's eta), some steps from host memory."""
    import torch
    d, K = 1_300_001, 4
    rng = np.random.default_rng(31)
    p = Pair(d, K, 0.9, 0.2, ratio=0.001, seed=2, variant=variant)
    for t in range(5):
        eta = 0.2 * 0.5 * (1 + np.cos(np.pi * t / 8))
        p.gpu.set_eta(eta)
        p.ref.set_eta(eta)
        g = _grads(rng, K, d)
        if t % 2:
            p.gpu.step_host(torch.from_numpy(g).pin_memory())
            r = p.ref.step(g)
        else:
            r = p.step(g)
        p.compare(r, residuals=(t == 4))
    p.compare_stats()
    assert p.gpu.check() == 0


def test_server_momentum_moves_coordinates_off_the_union():
    """Alg. 3's server momentum keeps moving every coordinate that moved
    before, so w changes off the step's union: the counter of changed
    coordinates (the RCC numerator) exceeds the union count."""
    d, K = 200_003, 2
    rng = np.random.default_rng(32)
    p = Pair(d, K, 0.9, 0.1, ratio=0.001, seed=1, variant="server_momentum")
    for t in range(4):
        r = p.step(_grads(rng, K, d))
        p.compare(r)
    s = p.compare_stats()
    assert s["changed"] > s["union"]


@pytest.mark.parametrize("variant", ["local_momentum", "local_momentum_mfm"])
def test_local_momentum_detach(variant):
    """The DEF-A-like detached points of the local-momentum baseline,
    w_{t,k} = w_t - lambda e_{t,k}, written by the step."""
    import torch
    d, K = 1_300_001, 3
    rng = np.random.default_rng(33)
    p = Pair(d, K, 0.9, 0.1, ratio=0.002, seed=4, variant=variant, lam=0.3)
    out = torch.empty((K, d), dtype=torch.float32, device=p.dev)
    p.gpu.set_detach_output(out)
    for t in range(3):
        r = p.step(_grads(rng, K, d))
        p.compare(r)
        torch.cuda.synchronize()
        for k in range(K):
            np.testing.assert_array_equal(out[k].cpu().numpy().view(np.uint32),
                                          p.ref.worker_params(k).view(np.uint32))
    p.compare_stats()


def test_variant_refusals():
    from paper_1905_12948_gb300 import GMC
    from paper_1905_12948_gb300.gmc import GMCError
    import torch
    with pytest.raises(GMCError):
        GMC(1000, 2, 0.9, 0.1, compressor="rbgs", ratio=0.1, block=10, variant="lr_in_residual")
    with pytest.raises(GMCError):
        GMC(1000, 2, 0.9, 0.1, lam=0.5, variant="server_momentum")
    g = GMC(1000, 2, 0.9, 0.1, variant="lr_in_residual")
    with pytest.raises(GMCError):
        g.set_lambda(0.5)
    g.set_params(torch.zeros(1000, device="cuda"))
    g.step(torch.ones((2, 1000), device="cuda"))
    assert g.lib.gmc_set_variant(g.h, 0) == 5  # GMC_ESTATE: after a step
    g.set_params(torch.zeros(1000, device="cuda"))
    assert g.lib.gmc_set_variant(g.h, 1) == 0  # allowed again before the first step
