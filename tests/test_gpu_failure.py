"""Failure detection without a GPU fault.

* A bounded wait that runs out: the test hook withholds one item's copy in a
  bulk pass, so the waits on it give up after a short limit; the kernel
  returns, gmc_check reports GMC_ETIMEOUT, and a reset (or a new handle) steps
  exactly as the oracle again.
* A device allocation that fails: the allocation hook makes the n-th
  allocation of gmc_create / gmc_set_variant fail as cudaMalloc does when
  memory runs out; the call returns GMC_ENOMEM, leaks nothing, and leaves an
  existing handle as it was.
"""
import ctypes
import gc

import numpy as np
import pytest

from parity_util import Pair

pytestmark = pytest.mark.gpu

GMC_OK, GMC_EINVAL, GMC_ENOMEM, GMC_ETIMEOUT = 0, 1, 2, 8
TILE = 4096


def _lib():
    from paper_1905_12948_gb300 import gmc
    return gmc.load()


def _grads(rng, K, d):
    return (rng.standard_normal((K, d)) * 0.1).astype(np.float32)


@pytest.mark.parametrize("compressor,d,K,hold", [
    ("topk", 1_300_001, 3, (5, 1)),      # bulk top-k pass (d >= 4096 * 2 * SMs), an odd worker
    ("topk", 1_300_001, 4, (0, 0)),      # the first fixed tile of CTA 0, the lead warps' worker
    ("topk_approx", 1_300_001, 2, (317, 1)),  # the last tile, ragged
    ("rbgs", 700_001, 3, (40, 2)),       # bulk RBGS pass (d >= 4096 * SMs)
])
def test_withheld_copy_times_out_and_is_reported(compressor, d, K, hold):
    import torch
    lib = _lib()
    rng = np.random.default_rng(11)
    ratio = 0.05 if compressor == "rbgs" else 0.001
    p = Pair(d, K, 0.9, 0.1, compressor=compressor, ratio=ratio, block=4096, seed=3)
    for _ in range(2):
        r = p.step(_grads(rng, K, d))
    p.compare(r)
    assert p.gpu.check() == GMC_OK
    tile, k = hold
    assert lib.gmc_test_withhold_copy(p.gpu.h, tile, k, 50_000_000) == GMC_OK
    g = torch.from_numpy(_grads(rng, K, d)).cuda()
    p.gpu.step(g)
    torch.cuda.synchronize()
    st = p.gpu.check()
    assert st == GMC_ETIMEOUT, lib.gmc_strerror(st)
    assert b"bounded wait" in lib.gmc_strerror(GMC_ETIMEOUT)
    assert p.gpu.check() == GMC_ETIMEOUT  # reading does not clear it

    # the same handle after a reset, and a new handle, step as the oracle does
    p2 = Pair(d, K, 0.9, 0.1, compressor=compressor, ratio=ratio, block=4096, seed=3)
    w0 = (np.random.default_rng(5).standard_normal(d) * 0.01).astype(np.float32)
    p.gpu.set_params(torch.from_numpy(w0).cuda())
    p.ref.set_params(w0)
    p2.gpu.set_params(torch.from_numpy(w0).cuda())
    p2.ref.set_params(w0)
    assert p.gpu.check() == GMC_OK
    for _ in range(3):
        g = _grads(rng, K, d)
        r = p.step(g)
        r2 = p2.step(g)
    p.compare(r)
    p2.compare(r2)
    assert p.gpu.check() == GMC_OK and p2.gpu.check() == GMC_OK
    p.gpu.close()
    p2.gpu.close()


def test_withhold_refused_without_a_bulk_pass():
    import torch
    from paper_1905_12948_gb300 import GMC
    lib = _lib()
    small = GMC(100_000, 2, 0.9, 0.1, compressor="topk", ratio=0.01)  # load/store pass
    small.set_params(torch.zeros(100_000, device="cuda"))
    assert lib.gmc_test_withhold_copy(small.h, 0, 0, 1_000_000) == GMC_EINVAL
    small.close()
    big = GMC(1_300_001, 2, 0.9, 0.1, compressor="topk", ratio=0.001)
    assert lib.gmc_test_withhold_copy(big.h, 0, 2, 1_000_000) == GMC_EINVAL   # worker out of range
    assert lib.gmc_test_withhold_copy(big.h, 318, 0, 1_000_000) == GMC_EINVAL  # tile out of range
    assert lib.gmc_test_withhold_copy(big.h, 0, 0, 0) == GMC_EINVAL            # no limit
    assert lib.gmc_test_withhold_copy(big.h, 0, 0, 3_000_000_000) == GMC_EINVAL
    big.close()


@pytest.mark.parametrize("d,K,compressor", [
    (100_000, 4, 0),      # top-k, load/store pass
    (1_300_001, 3, 0),    # top-k, bulk pass (candidate regions per CTA)
    (700_001, 5, 1),      # RBGS
    (300_000, 2, 2),      # approximate top-s
])
def test_create_allocation_failures_leak_nothing(d, K, compressor):
    import torch
    lib = _lib()
    torch.cuda.init()
    gc.collect()  # handles of earlier tests still waiting for the collector
    live0 = lib.gmc_test_fail_alloc(-1)
    failures = 0
    for i in range(64):
        lib.gmc_test_fail_alloc(i)
        h = ctypes.c_void_p()
        st = lib.gmc_create(ctypes.byref(h), d, K, 0.9, 0.1, compressor, 0.01, 4096)
        live = lib.gmc_test_fail_alloc(-1)
        if st == GMC_OK:
            assert live > live0
            lib.gmc_destroy(h)
            break
        assert st == GMC_ENOMEM, (i, st)
        assert h.value is None
        assert live == live0, f"allocation {i} failed and {live - live0} allocations leaked"
        failures += 1
    else:
        pytest.fail("gmc_create never succeeded")
    assert failures >= 8  # every allocation of the handle's state was made to fail once
    assert lib.gmc_test_fail_alloc(-1) == live0


def test_set_variant_allocation_failure_leaves_the_handle_usable():
    import torch
    lib = _lib()
    d, K = 200_003, 3
    rng = np.random.default_rng(4)
    gc.collect()
    p = Pair(d, K, 0.9, 0.1, compressor="topk", ratio=0.01)
    live = lib.gmc_test_fail_alloc(-1)
    for variant in (1, 3):  # Alg. 3's server momentum, the local momentum: one allocation each
        lib.gmc_test_fail_alloc(0)
        assert lib.gmc_set_variant(p.gpu.h, variant) == GMC_ENOMEM
        assert lib.gmc_test_fail_alloc(-1) == live
    for _ in range(3):  # still Alg. 1, still exact
        r = p.step(_grads(rng, K, d))
    p.compare(r)
    p.compare_stats()
    assert p.gpu.check() == GMC_OK
    p.gpu.close()
    assert lib.gmc_test_fail_alloc(-1) == live - _handle_allocations(d, K)


def _handle_allocations(d, K):
    """Device allocations one top-k handle of this size holds (counted with the hook)."""
    lib = _lib()
    before = lib.gmc_test_fail_alloc(-1)
    h = ctypes.c_void_p()
    assert lib.gmc_create(ctypes.byref(h), d, K, 0.9, 0.1, 0, 0.01, 4096) == GMC_OK
    n = lib.gmc_test_fail_alloc(-1) - before
    lib.gmc_destroy(h)
    assert lib.gmc_test_fail_alloc(-1) == before
    return n
