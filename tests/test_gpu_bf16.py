"""bfloat16 gradient input (gmc_step_bf16 / gmc_step_host_bf16): the step on
bf16 rows equals the oracle's step on the same values widened to fp32, for
every compressor, both dense passes, every row alignment (odd d, a pointer
one element past an aligned address), deferred aggregation, a variant with
its own state, and host memory (page-locked and pageable)."""
import numpy as np
import pytest

from parity_util import Pair

pytestmark = pytest.mark.gpu


def _bf16_grads(rng, K, d, dev, offset=0):
    """bf16 gradients on the device (optionally offset by `offset` elements
    from an aligned allocation) and their exact fp32 values for the oracle."""
    import torch
    g = torch.from_numpy((rng.standard_normal((K, d)) * np.exp(rng.uniform(-3, 0, size=d)))
                         .astype(np.float32)).to(torch.bfloat16)
    buf = torch.empty(K * d + offset, dtype=torch.bfloat16, device=dev)
    view = buf[offset:].view(K, d)
    view.copy_(g.to(dev))
    return view, g.float().numpy()


CASES = [
    dict(compressor="topk", d=1_300_001, K=4, ratio=0.002),
    dict(compressor="topk", d=1_300_001, K=6, ratio=0.002),
    dict(compressor="topk", d=1_300_001, K=3, ratio=0.002, offset=1),
    dict(compressor="topk", d=50_003, K=3, ratio=0.01),
    dict(compressor="topk_approx", d=1_300_001, K=3, ratio=1 / 1024),
    dict(compressor="rbgs", d=4096 * 160 + 3, K=5, ratio=0.05, block=4096, lam=0.5),
    dict(compressor="rbgs", d=4096 * 160 + 3, K=2, ratio=0.05, block=4096, lam=0.5, offset=3),
    dict(compressor="rbgs", d=70_001, K=3, ratio=0.1, block=1000, lam=0.5),
    dict(compressor="topk", d=1_300_001, K=3, ratio=0.002, variant="local_momentum"),
    dict(compressor="topk", d=50_003, K=2, ratio=0.01, variant="lr_in_residual"),
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: "-".join(str(v) for v in c.values()))
def test_bf16_step_parity(case):
    case = dict(case)
    d, K = case.pop("d"), case.pop("K")
    offset = case.pop("offset", 0)
    rng = np.random.default_rng(d + K + offset)
    p = Pair(d, K, 0.9, 0.1, seed=21, **case)
    for t in range(4):
        g_dev, g = _bf16_grads(rng, K, d, p.dev, offset)
        r = p.step(g, grads_dev=g_dev)
        p.compare(r, state=(t == 3 or case["compressor"] == "rbgs"))
    p.compare_stats()
    assert p.gpu.check() == 0


@pytest.mark.parametrize("pinned", [True, False])
def test_bf16_host_steps(pinned):
    import torch
    d, K = 1_300_001, 3
    rng = np.random.default_rng(7)
    p = Pair(d, K, 0.9, 0.1, ratio=0.002, seed=3)
    for t in range(3):
        g_dev, g = _bf16_grads(rng, K, d, p.dev)
        host = g_dev.cpu()
        if pinned:
            host = host.pin_memory()
        p.gpu.step_host(host)
        r = p.ref.step(g)
        p.compare(r)
    p.compare_stats()
    assert p.gpu.check() == 0


def test_bf16_misaligned_pointer_refused():
    import torch
    from paper_1905_12948_gb300 import GMC
    g = GMC(1000, 2, 0.9, 0.1, ratio=0.01)
    g.set_params(torch.zeros(1000, device="cuda"))
    buf = torch.zeros(2 * 1000 + 1, dtype=torch.bfloat16, device="cuda")
    assert g.lib.gmc_step_bf16(g.h, buf.data_ptr() + 1, None) == 1  # GMC_EINVAL: odd address
    assert g.lib.gmc_step_bf16(g.h, buf.data_ptr(), None) == 0
