"""gmc_topk_noalloc against the regular top-k path.

Some callers cannot allocate device memory: for example code whose device
memory is all owned by another allocator, such as a framework's caching pool
or a serving process with a fixed memory budget. gmc_topk_noalloc gives them
the library's top-k compressor with its scratch in a fixed array inside the
library, so neither the library nor the caller allocates anything per call.

This test calls it through the C ABI and checks that it keeps the same
coordinates and values as the regular entry point (gmc_step of a handle with
one worker, beta = 0 and a zero state, whose accumulator is then exactly the
input vector), on two calls in a row with different inputs and sizes, so the
second call also shows that the shared scratch is reset between calls.
"""
import ctypes

import numpy as np
import pytest

from parity_util import ATOL, RTOL

pytestmark = pytest.mark.gpu

GMC_ETOOBIG = 7


def _regular_topk(x, k):
    """Top-k of x through gmc_step + gmc_get_selected (the existing path)."""
    import torch
    from paper_1905_12948_gb300 import GMC
    n = x.numel()
    ratio = (k + 0.5) / n  # k = floor(ratio * n)
    h = GMC(n, 1, beta=0.0, eta=1.0, compressor="topk", ratio=ratio, device=x.device)
    h.set_params(torch.zeros(n, dtype=torch.float32, device=x.device))
    h.step(x.view(1, n))
    idx, val = h.selected(0)
    assert h.check() == 0
    h.close()
    return idx.cpu().numpy(), val.cpu().numpy()


def _noalloc_topk(lib, x, k):
    import torch
    n = x.numel()
    idx = torch.empty(k, dtype=torch.int32, device=x.device)
    val = torch.empty(k, dtype=torch.float32, device=x.device)
    stream = torch.cuda.current_stream().cuda_stream
    st = lib.gmc_topk_noalloc(x.data_ptr(), n, k, idx.data_ptr(), val.data_ptr(), stream)
    assert st == 0, lib.gmc_strerror(st)
    torch.cuda.synchronize()
    return idx.cpu().numpy().astype(np.int64), val.cpu().numpy()


def test_noalloc_topk_matches_regular_path_twice():
    import torch
    from paper_1905_12948_gb300 import gmc
    lib = gmc.load()
    rng = np.random.default_rng(2024)
    dev = torch.device("cuda")
    cases = [(1_000_003, 1_000), (70_001, 700)]
    for n, k in cases:  # two calls in a row
        x_np = (rng.standard_normal(n) * np.exp(rng.uniform(-4, 0, size=n))).astype(np.float32)
        x_np[rng.integers(0, n, size=50)] = 0.5  # ties across tiles
        x = torch.from_numpy(x_np).to(dev)
        want_idx, want_val = _regular_topk(x, k)
        got_idx, got_val = _noalloc_topk(lib, x, k)
        np.testing.assert_array_equal(got_idx, want_idx)
        np.testing.assert_allclose(got_val, want_val, rtol=RTOL, atol=ATOL)


def test_noalloc_rejects_sizes_above_its_scratch():
    import torch
    from paper_1905_12948_gb300 import gmc
    lib = gmc.load()
    x = torch.zeros(4, dtype=torch.float32, device="cuda")
    out_i = torch.empty(4, dtype=torch.int32, device="cuda")
    out_v = torch.empty(4, dtype=torch.float32, device="cuda")
    assert lib.gmc_topk_noalloc(x.data_ptr(), (1 << 26) + 1, 4, out_i.data_ptr(),
                                out_v.data_ptr(), None) == GMC_ETOOBIG
    assert lib.gmc_topk_noalloc(x.data_ptr(), 4, 5, out_i.data_ptr(), out_v.data_ptr(), None) == 1
    assert b"2^26" in lib.gmc_strerror(GMC_ETOOBIG)
